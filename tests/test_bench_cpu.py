"""bench.py on the CPU: the reference arm's JSON line (the oracle timed on a bounded
sample) and the algorithmic FLOP / byte models behind the roofline figures."""

import json
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from synth import hero_inputs as hi  # noqa: E402


@pytest.mark.parametrize("workload", ["tiny_f32", "small_bf16_decoder"])
def test_reference_arm_prints_one_json_line(workload):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", workload, "--steps", "1", "--warmup", "3",
                        "--cpu-sample", "4"], capture_output=True, text=True, timeout=600,
                       cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "impl", "cpu_baseline", "e2e", "config"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["warmup"] >= 3
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]


def test_flop_model_of_the_stack():
    """4 I d FLOP per FFN token for gate/up, 2 I d for down, 2 d d_r per adapter token
    each way (the down projection folded into gate/up for bf16), 4 d 512 per token for
    the router contraction with its bf16 operand pair."""
    cfg = hi.CONFIGS["llama31_8b_prefill"]
    T, d, I, r, L = cfg.n_tokens, cfg.d_model, cfg.d_ff, cfg.d_r, cfg.n_layers
    counts = np.full(L, 12000)
    w = bench.algorithmic_work(cfg, counts, 2)
    na = T - 12000
    assert w["ffn_gate_up"] == pytest.approx(2 * L * (2.0 * 12000 * 2 * I * d + 2.0 * na * r * d))
    assert w["ffn_down"] == pytest.approx(2 * L * 2.0 * 12000 * I * d)
    assert w["adapter_up"] == pytest.approx(2 * L * 2.0 * na * d * r)
    assert w["router_gemm"] == pytest.approx(2 * L * 2.0 * T * 512 * 2 * d)
    assert "attn_core" not in w


def test_flop_and_byte_models_of_attention():
    """Causal attention: 4 hd (s + 1) FLOP per query head at position s, summed over the
    sequence; a decoding step reads every cached key and value once."""
    cfg = hi.CONFIGS["llama31_8b_decoder"]
    B, S, H, hd, L = cfg.batch, cfg.seq_len, cfg.n_heads, 128, cfg.n_layers
    w = bench.algorithmic_work(cfg, np.full(L, cfg.n_tokens), 1)
    assert w["attn_core"] == pytest.approx(L * B * H * sum(4.0 * hd * (s + 1) for s in range(S)))
    kv = hi.CONFIGS["llama31_8b_kvdecode"]
    nb = bench.algorithmic_bytes(kv, np.full(L, 50), 1)
    assert nb["attn_core"] == pytest.approx(L * kv.batch * kv.n_kv_heads * (kv.seq_len + 1) * hd * 2 * 2)
    # at 64 tokens the FFN classes are weight-bound: bytes at HBM outlast FLOPs at the tensor peak
    wk = bench.algorithmic_work(kv, np.full(L, 50), 1)
    assert nb["ffn_gate_up"] / 6.6e12 > wk["ffn_gate_up"] / 1.7e15


def test_workload_descriptions_name_the_shapes():
    assert "4x4096" in bench.workload_desc(hi.CONFIGS["llama31_8b_prefill"], 0.2687)
    desc = bench.workload_desc(hi.CONFIGS["llama31_8b_kvdecode"], 0.2687)
    assert "64 sequences" in desc and "position 4096" in desc and "H_kv=8" in desc


def test_gpus_flag_starts_its_own_ranks(monkeypatch):
    """--gpus N without an outside launcher re-runs bench.py as N ranks of one node under
    torch.distributed.run on a 127.0.0.1 rendezvous (no GPU is touched here)."""
    seen = {}

    def fake_call(cmd):
        seen["cmd"] = cmd
        return 0

    monkeypatch.setattr(bench.subprocess, "call", fake_call)
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    monkeypatch.setattr(sys, "argv", ["bench.py", "--gpus", "4", "--steps", "2"])
    assert bench.main() == 0
    cmd = seen["cmd"]
    assert cmd[1:3] == ["-m", "torch.distributed.run"]
    assert "--nproc-per-node=4" in cmd and "--master-addr=127.0.0.1" in cmd
    assert cmd[-4:] == ["--gpus", "4", "--steps", "2"]


@pytest.mark.parametrize("bypass", [0.0, 0.27, 0.39])
def test_bypass_sweep_points_have_a_committed_tau(bypass):
    """The Llama-2-13B sweep (0 / 27 / 39% bypass) selects a calibrated tau per point;
    tau grows with the budget (more tokens below it) and 0% admits every token."""
    tau = hi.calibrated_tau("llama2_13b_prefill", bypass)
    if bypass == 0.0:
        assert tau == 0.0
    assert hi.calibrated_tau("llama2_13b_prefill", 0.39) > hi.calibrated_tau("llama2_13b_prefill", 0.27)
