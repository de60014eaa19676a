"""Measure the oracle's own sensitivity of the gates to tiny input perturbations.

Usage: python tests/golden/gate_sensitivity.py [workload ...]   (minutes per workload)

With bf16 rounding at the precision contract's points (u, the SwiGLU product,
the adapter hidden, the router operand pair), a relative perturbation of h_0 as
small as fp32 arithmetic makes flips some roundings; the flips feed through the
residual stream into the next blocks' router inputs and the gate difference
grows with depth.  This script runs the float64 oracle twice per workload, on a
token sample the full-size GPU test compares (same tokens, same count), with h_0
and with h_0 (1 + eps N(0,1)) for eps = 1e-7, 3e-7 and 1e-6, under forced
all-FFN decisions, and records the largest gate and hidden state differences
per block.  The free-running GPU parity tests derive their
gate bound for deep stacks from these numbers; nothing here runs the CUDA path.
"""

from __future__ import annotations

import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import hero_oracle as ho  # noqa: E402
from synth import hero_inputs as hi  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "gate_sensitivity.json")
# tokens per workload: the sample sizes of the full-size sampled GPU tests
SAMPLE = {"small_bf16": 32, "llama2_7b_prefill": 64, "llama31_8b_prefill": 64,
          "llama31_8b_decode": 64, "llama2_13b_prefill": 32, "llama31_8b_paper": 32}
EPS = (1e-7, 3e-7, 1e-6)


def measure(name: str, bypass=None):
    cfg = hi.CONFIGS[name]
    tau = hi.calibrated_tau(name, bypass)
    w = hi.generate_weights(cfg)
    rows = hi.sample_tokens(cfg.n_tokens, SAMPLE[name])
    h = hi.generate_h_in(cfg)[rows].astype(np.float64)
    P = hi.generate_attn_delta(cfg)[:, rows]
    oc = ho.OracleConfig.from_stack(cfg)
    ones = np.ones((cfg.n_layers, len(rows)), np.uint8)
    base = ho.routed_ffn_stack(oc, w, h, P, tau, mode="force", mask_in=ones)
    rng = np.random.default_rng(0)
    out = {"sample": int(len(rows)), "layers": cfg.n_layers}
    for eps in EPS:
        pert = ho.routed_ffn_stack(oc, w, h * (1.0 + eps * rng.standard_normal(h.shape)), P, tau,
                                   mode="force", mask_in=ones)
        dg = np.abs(pert["gate"] - base["gate"]).max(axis=1)
        dh = np.max(np.abs(pert["h_out"] - base["h_out"]), axis=1) / np.max(np.abs(base["h_out"]), axis=1)
        out[f"{eps:.0e}"] = {"gate_max": float(dg.max()), "h_rel_max": float(dh.max()),
                             "gate_by_block": [float(x) for x in dg]}
    return out


def main():
    names = sys.argv[1:] or ["small_bf16", "llama2_7b_prefill", "llama31_8b_prefill",
                             "llama31_8b_decode", "llama2_13b_prefill"]
    table = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            table = json.load(f)
    for n in names:
        res = measure(n, 0.27 if n == "llama2_13b_prefill" else None)
        table[n] = res
        print(n, {k: v["gate_max"] for k, v in res.items() if isinstance(v, dict)}, flush=True)
        with open(OUT, "w") as f:
            json.dump(table, f, indent=1, sort_keys=True)


if __name__ == "__main__":
    main()
