"""Calibrate the execution threshold tau_exec of each workload to its bypass budget.

Usage: python synth/calibrate_tau.py [workload ...] [--sample N]

The paper reaches its budgets by training (alpha_t, Sec. 3.3); with random-init
routers this build instead bisects one shared tau_exec per workload so that the
oracle's free-running bypass fraction (adapter executions / (L_R T)) matches the
target.  Large workloads use a fixed evenly spread token sample (tokens are
independent through the stack); decoder workloads (real attention) use the same
causal prefix of every sequence.  The result is written to synth/tau.json and is
read by both the CUDA harness and the tests; nothing here runs the CUDA path.
"""

from __future__ import annotations

import argparse
import json
import os
import sys
import time

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from synth import hero_inputs as hi  # noqa: E402
from oracle import hero_oracle as ho  # noqa: E402

TAU_FILE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "tau.json")


def _bypass(cfg, w, h, P, tau, attn=None):
    oc = ho.OracleConfig.from_stack(cfg)
    if attn is None:
        r = ho.routed_ffn_stack(oc, w, h, P, tau)
    else:
        wa, n_seqs, seq_len = attn
        r = ho.decoder_forward(oc, w, wa, h, tau, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta,
                               n_seqs, seq_len)
    return ho.bypass_fraction(r["mask"], cfg.n_dense), r


def _decoder_sample(cfg, sample):
    """Token sample of a decoder workload: attention couples the tokens of a sequence,
    so the sample is the same causal prefix of every sequence (a prefix of a causal
    decoder's input is computed exactly without the rest of its sequence)."""
    prefix = max(1, min(cfg.seq_len, sample // cfg.batch))
    idx = (np.arange(cfg.batch)[:, None] * cfg.seq_len + np.arange(prefix)[None, :]).reshape(-1)
    return idx, prefix


def calibrate(cfg, target, sample, iters=14):
    t0 = time.time()
    w = hi.generate_weights(cfg)
    attn = None
    if cfg.n_heads:
        idx, prefix = _decoder_sample(cfg, sample)
        attn = (hi.generate_attn_weights(cfg), cfg.batch, prefix)
        P = None
    else:
        idx = hi.sample_tokens(cfg.n_tokens, sample)
        P = hi.generate_attn_delta(cfg)[:, idx]
    h = hi.generate_h_in(cfg)[idx]
    n_dec = (cfg.n_layers - cfg.n_dense) * len(idx)     # routed decisions
    if target <= 0.0:
        return {"tau": 0.0, "bypass": 0.0, "sample": int(len(idx)), "decisions": n_dec}
    lo, hi_ = 0.0, 1.0        # bypass(lo) = 0 (every g >= 0), bypass(hi) = 1
    best = None
    for _ in range(iters):
        mid = 0.5 * (lo + hi_)
        b, _ = _bypass(cfg, w, h, P, mid, attn)
        if best is None or abs(b - target) < abs(best[1] - target):
            best = (mid, b)
        if abs(b - target) * n_dec < 0.5:
            break
        if b < target:
            lo = mid
        else:
            hi_ = mid
        print(f"  {cfg.name}: tau={mid:.6f} bypass={b:.4f} ({time.time() - t0:.0f}s)", flush=True)
    tau, b = best
    res = {"tau": tau, "bypass": b, "sample": int(len(idx)), "decisions": n_dec, "target": target}
    if attn is not None:
        res["prefix"] = int(attn[2])
    return res


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("names", nargs="*")
    ap.add_argument("--sample", type=int, default=256)
    args = ap.parse_args()
    names = args.names or list(hi.CONFIGS)
    table = {"note": "tau_exec per workload@bypass, bisected on the float64 oracle "
                     "(synth/calibrate_tau.py) over the stated token sample",
             "tau": {}}
    if os.path.exists(TAU_FILE):
        with open(TAU_FILE) as f:
            table = json.load(f)
    for name in names:
        cfg = hi.CONFIGS[name]
        if cfg.kv_decode_of:   # uses its prefill workload's tau
            continue
        targets = hi.BYPASS_SWEEP_13B if name == "llama2_13b_prefill" else (cfg.bypass,)
        for tgt in targets:
            res = calibrate(cfg, tgt, args.sample)
            table["tau"][f"{name}@{tgt:.4f}"] = res
            print(name, tgt, res, flush=True)
            with open(TAU_FILE, "w") as f:
                json.dump(table, f, indent=1, sort_keys=True)


if __name__ == "__main__":
    main()
