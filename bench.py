"""Throughput of the routed FFN stack on GB300 (one JSON line on rank 0).

python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                [--workload NAME] [--bypass B] [--cpu-sample N] [--no-cpu-baseline]

A step is one pass of the whole routed FFN stack (all routed blocks: memory
readout, router score, compaction, FFN / adapter, scatter into the residual,
memory update) over the workload's T tokens.  Inputs (weights 11.3 GB, the
attention stand-in 4.3 GB) are far larger than the 129 MB L2, so no flush is
needed between steps.  With N > 1 ranks (torchrun), every rank runs its own
token shard of the same size on its own GPU (weak scaling, no collective on the
data path); value = all ranks' tokens / the slowest rank's time.  Without an outside
launcher, --gpus N > 1 starts the N ranks itself (torch.distributed.run).

Decoder workloads (--workload llama31_8b_decoder, small_bf16_decoder) run the full
decoder forward instead: every block's h_bar comes from the real attention
sublayer (Eq. 1) rather than the stand-in; a step is all blocks' attention plus
routed FFN over B sequences of S tokens.  The KV-cache decoding workload
(llama31_8b_kvdecode) first fills the cache of 64 sequences with 4096-token
prefills (untimed); a step is then one new token for each sequence at position
4096 (every step decodes the same position: the context stays 4096).

--impl reference times the CPU oracle (the only reference this method has) on a
bounded token sample per step, on rank 0 only (decoder workloads: a causal prefix
of one sequence, which the oracle computes exactly without the rest).
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synth import hero_inputs as hi  # noqa: E402

METRIC = "routed-FFN-stack tokens/s at Llama-3.1-8B shapes; % of bf16 tensor peak"
# decoder workloads: the same tokens/s, with the attention sublayers inside the step
METRIC_DECODER = "decoder-forward (attention + routed FFN) tokens/s at Llama-3.1-8B shapes"
METRIC_KVDECODE = "KV-cache decoding tokens/s (attention over the cache + routed FFN) at Llama-3.1-8B shapes"


def metric_for(cfg):
    if cfg.kv_decode_of:
        return METRIC_KVDECODE
    return METRIC_DECODER if cfg.n_heads else METRIC
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# DRAM bytes (read + write) per launch of the dominant kernel at the default workload,
# taken from a single-kernel ncu capture of a smaller case of the same kernel and scaled
# to the full launch by the FFN rows it processes; reported only for the unmodified
# default workload, and emptied whenever the kernel changes before it is captured again.
# (Empty: the last capture, 2942 MB per launch, predates later edits of the GEMM kernel.)
DOMINANT_TRAFFIC = {}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def workload_desc(cfg, bypass):
    blocks = (f"{cfg.n_layers} routed blocks" if not cfg.n_dense else
              f"{cfg.n_dense} dense + {cfg.n_layers - cfg.n_dense} routed blocks")
    variant = f", router ablation bits {cfg.router_variant}" if cfg.router_variant else ""
    if cfg.n_heads:
        variant += (f", causal attention H={cfg.n_heads}, H_kv={cfg.n_kv_heads}, hd=128, "
                    f"RoPE theta={cfg.rope_theta:g}")
    shape = (f"T={cfg.n_tokens} per step ({cfg.batch} sequences, one new token each at position "
             f"{cfg.seq_len} after a {cfg.seq_len}-token cached prefix)" if cfg.kv_decode_of else
             f"T={cfg.n_tokens} ({cfg.batch}x{cfg.seq_len})")
    return (f"{cfg.name}: {blocks}, d={cfg.d_model}, I={cfg.d_ff}, "
            f"d_r={cfg.d_r}, d_m={cfg.d_m}, {shape}, "
            f"{cfg.dtype}, bypass target {bypass:.2%}{variant}, random-init weights, seeded inputs")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={','.join(self.FIELDS)}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def algorithmic_work(cfg, counts_per_step, steps, routed=True):
    """Algorithmic FLOPs per kernel class over the timed steps (counts: FFN tokens per
    block).  bf16 models run the adapter's down projection inside the FFN gate/up
    launch of the same block (grouped), so that class carries its FLOPs too."""
    T, d, I, r = cfg.n_tokens, cfg.d_model, cfg.d_ff, cfg.d_r
    nY = cfg.d_enc + cfg.d_head
    k_r = 2 * d if cfg.dtype == "bf16" else d   # bf16: the operand pair [hi | lo]
    nf = np.asarray(counts_per_step, dtype=np.float64)
    na = T - nf
    work = {
        "ffn_gate_up": steps * float(np.sum(2.0 * nf * 2 * I * d)),
        "ffn_down": steps * float(np.sum(2.0 * nf * I * d)),
        "router_gemm": steps * float((cfg.n_layers - cfg.n_dense) * 2.0 * T * nY * k_r)
        if routed else 0.0,
        "adapter_down": steps * float(np.sum(2.0 * na * r * d)),
        "adapter_up": steps * float(np.sum(2.0 * na * d * r)),
    }
    if cfg.dtype == "bf16":
        work["ffn_gate_up"] += work.pop("adapter_down")
    if cfg.n_heads:   # decoder: projections and causal attention of every block
        hd = cfg.d_model // cfg.n_heads
        nqkv = (cfg.n_heads + 2 * cfg.n_kv_heads) * hd
        B, S = cfg.batch, cfg.seq_len
        work["attn_proj"] = steps * cfg.n_layers * 2.0 * T * d * (nqkv + cfg.n_heads * hd)
        if cfg.kv_decode_of:   # one query per sequence over S + 1 keys
            work["attn_core"] = steps * cfg.n_layers * B * cfg.n_heads * 4.0 * hd * (S + 1)
        else:   # q k^T and p v over the causal triangle (S (S + 1) / 2 scores per head)
            work["attn_core"] = steps * cfg.n_layers * B * cfg.n_heads * 4.0 * hd * S * (S + 1) / 2
    return work


def algorithmic_bytes(cfg, counts_per_step, steps):
    """Algorithmic HBM bytes per kernel class over the timed steps: every weight a
    class multiplies is read once per block that runs it (bf16), and decoding
    attention reads the cached keys and values once.  Activations are left out
    (a lower bound; they matter only where the tensor bound wins anyway)."""
    d, I, r, L = cfg.d_model, cfg.d_ff, cfg.d_r, cfg.n_layers
    nf = np.asarray(counts_per_step)
    T = cfg.n_tokens
    nY = cfg.d_enc + cfg.d_head
    wb = 2.0
    out = {
        "ffn_gate_up": steps * wb * float(np.sum((nf > 0) * 2 * I * d + (nf < T) * r * d)),
        "ffn_down": steps * wb * float(np.sum((nf > 0) * I * d)),
        "router_gemm": steps * wb * (L - cfg.n_dense) * nY * 2 * d,
        "adapter_up": steps * wb * float(np.sum((nf < T) * d * r)),
    }
    if cfg.n_heads:
        hd = d // cfg.n_heads
        nqkv = (cfg.n_heads + 2 * cfg.n_kv_heads) * hd
        out["attn_proj"] = steps * wb * L * (nqkv + cfg.n_heads * hd) * d
        if cfg.kv_decode_of:
            out["attn_core"] = steps * wb * L * cfg.batch * cfg.n_kv_heads * (cfg.seq_len + 1) * hd * 2
    return out


def oracle_step(ho, cfg, w, h_np, tau, n_sample, P_np=None):
    """One oracle pass over a bounded sample of the workload: evenly spread tokens of
    the stack (tokens are independent), or the first n_sample positions of sequence 1
    of a decoder workload (a causal prefix needs nothing after it)."""
    oc = ho.OracleConfig.from_stack(cfg)
    if cfg.n_heads:
        wa = hi.generate_attn_weights(cfg)
        n = min(n_sample, cfg.seq_len)
        rows = np.arange(n)
        h = h_np[rows]

        def step():
            ho.decoder_forward(oc, w, wa, h, tau, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta, 1, n)
        return step, rows, (f"positions 0..{n - 1} of sequence 1 (of {cfg.batch}x{cfg.seq_len}) "
                            f"through all {cfg.n_layers} blocks with attention, float64 numpy")
    rows = hi.sample_tokens(cfg.n_tokens, n_sample)
    h = h_np[rows]
    P = (hi.generate_attn_delta(cfg) if P_np is None else P_np)[:, rows]

    def step():
        ho.routed_ffn_stack(oc, w, h, P, tau)
    return step, rows, (f"{len(rows)} evenly spread tokens of T={cfg.n_tokens} through all "
                        f"{cfg.n_layers} blocks, float64 numpy")


def reference_arm(args, rank, world):
    if rank != 0:
        return
    from oracle import hero_oracle as ho
    cfg = hi.CONFIGS[args.workload]
    if args.bypass is not None:
        cfg = cfg.replace(bypass=args.bypass)
    tau = hi.calibrated_tau(cfg.name, args.bypass)
    w = hi.generate_weights(cfg)
    step, rows, sample = oracle_step(ho, cfg, w, hi.generate_h_in(cfg), tau, args.cpu_sample)
    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    v = len(rows) * args.steps / dt
    cores = len(os.sched_getaffinity(0))
    line = {"metric": metric_for(cfg), "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": workload_desc(cfg, cfg.bypass), "sample": sample},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{len(rows)} tokens x {cfg.n_layers} blocks per step"},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def backward_flops(cfg, counts):
    """Algorithmic FLOPs of the training path's block backwards (decisions fixed): per FFN
    token the gate/up recomputation (4 I d), e = G W_down (2 I d) and du = [dgate|dup]
    [W_gate|W_up] (4 I d); per adapter token W_1 u, G W_2, da W_1 and the two weight
    gradients (2 d d_r each)."""
    T, d, I, r = cfg.n_tokens, cfg.d_model, cfg.d_ff, cfg.d_r
    nf = np.asarray(counts, dtype=np.float64)[cfg.n_dense:]
    return {"backward_gemm": float(np.sum(10.0 * nf * I * d + 6.0 * (T - nf) * d * r)),
            "wgrad": float(np.sum(4.0 * (T - nf) * d * r))}


def backward_arm(args, cfg, stack, hero, h, P, tau, stream, dev, world, rank, timed, sampler, t_gen):
    """Training-path step: the backward of every routed block's branch part (Sec. 3.1,
    Sec. 3.3) over the workload's T tokens, with the gates and decisions of one forward
    pass fixed, a seeded upstream gradient G and h_bar = the stack's input (the cost does
    not depend on the values).  Metric: tokens per second of one such pass."""
    import torch
    T, d, L, r = cfg.n_tokens, cfg.d_model, cfg.n_layers, cfg.d_r
    _, gate, mask, counts = stack(h, P, tau)
    torch.cuda.synchronize()
    stack.backward_init()
    G = torch.randn((T, d), device=dev, generator=torch.Generator(device=dev).manual_seed(3))
    gh = torch.empty((T, d), device=dev)
    gg = torch.empty((L, T), device=dev)
    g1 = torch.empty((L, r, d), device=dev)
    g2 = torch.empty((L, d, r), device=dev)
    blocks = range(cfg.n_dense + 1, L + 1)

    def step():
        for j in blocks:
            hero.hero_routed_block_backward(stack.model, j, T, h.data_ptr(), gate[j - 1].data_ptr(),
                                            mask[j - 1].data_ptr(), G.data_ptr(), 0, gh.data_ptr(),
                                            gg[j - 1].data_ptr(), g1[j - 1].data_ptr(),
                                            g2[j - 1].data_ptr(), stream.cuda_stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    stack.check()
    ms, clocks = timed(step, args.steps, sampler)
    stack.check()
    hero.hero_get_profile(stack.model, reset=True)
    hero.hero_set_profiling(stack.model, True)
    timed(step, args.steps)
    hero.hero_set_profiling(stack.model, False)
    prof = hero.hero_get_profile(stack.model, reset=True)
    stack.check()
    cnt = counts.cpu().numpy().astype(np.int64)
    work = backward_flops(cfg, cnt)
    peaks, peak_src = load_peaks()
    peak_tf = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    bms, bn = prof["backward_gemm"]
    achieved = work["backward_gemm"] * args.steps / (bms / 1e3) / 1e12 if bms else None
    value = world * T * args.steps / (ms / 1e3)
    line = {
        "metric": "routed-block backward (decisions fixed) tokens/s at the workload's shapes",
        "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
        "config": {"workload": workload_desc(cfg, cfg.bypass) + "; backward of every routed block",
                   "l2": "inputs larger than L2 (no flush): weights stream from HBM each block"},
        "roofline": {"kernel": "backward_gemm", "bound": "tensor", "achieved": achieved,
                     "peak": peak_tf, "unit": "TFLOP/s",
                     "frac": achieved / peak_tf if achieved else None, "traffic": None,
                     "peak_source": f"{peak_src} bf16_tflops_sustained",
                     "avg_launch_ms": bms / max(bn, 1)},
        "gpu_launches": int(sum(n for _, n in prof.values())),
        "clocks": clocks, "bypass": 1.0 - cnt[cfg.n_dense:].sum() / ((L - cfg.n_dense) * T),
        "ffn_counts": cnt.tolist(),
        "kernel_ms_per_step": {k: v[0] / args.steps for k, v in prof.items() if v[1]},
        "setup_s": {"generate": t_gen},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    stack.close()
    return 0


def launch_ranks(n: int) -> int:
    """--gpus N without an outside launcher: run this script again as N ranks of one node
    under torch.distributed.run (127.0.0.1 rendezvous on a free port); rank 0 prints."""
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.abspath(__file__),
           *sys.argv[1:]]
    return subprocess.call(cmd)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama31_8b_prefill", choices=sorted(hi.CONFIGS))
    ap.add_argument("--cpu-sample", type=int, default=8)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-dense", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-speculate", action="store_true",
                    help="batches of one 128-row tile: FFN on the routed tokens only, after the "
                         "router (default: every token, beside the router)")
    # overrides for profiling small cases (a line produced with them is not the workload's)
    ap.add_argument("--tau", type=float, default=None)
    ap.add_argument("--tokens", type=int, default=None)
    ap.add_argument("--layers", type=int, default=None)
    ap.add_argument("--router-variant", type=int, default=0,
                    help="Sec. 4.4 router ablation bits (1 history, 2 memread, 4 aux, 8 pos)")
    ap.add_argument("--d-m", type=int, default=None, help="memory width override (ablation)")
    ap.add_argument("--graph", action="store_true",
                    help="time CUDA-graph replays of one captured step (launch-bound decode)")
    ap.add_argument("--backward", action="store_true",
                    help="time the training path instead: every routed block's backward with "
                         "the decisions of one forward pass fixed")
    ap.add_argument("--bypass", type=float, default=None,
                    help="bypass target whose committed tau to use (e.g. 0, 0.27, 0.39 for "
                         "llama2_13b_prefill); default: the workload's own")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    if "WORLD_SIZE" not in os.environ and args.gpus > 1 and args.impl == "ours":
        return launch_ranks(args.gpus)
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and args.gpus != world:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={world}")
    if args.impl == "reference":
        return reference_arm(args, rank, world)

    import torch
    from paper_2609_08189_gb300 import build, hero

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if rank == 0:
        build.build()
    if dist:
        dist.barrier()
    hero.load()

    cfg = hi.CONFIGS[args.workload]
    if args.bypass is not None:
        cfg = cfg.replace(bypass=args.bypass)
    tau = hi.calibrated_tau(cfg.name, args.bypass) if args.tau is None else args.tau
    if args.tokens or args.layers:
        cfg = cfg.replace(n_tokens=args.tokens or cfg.n_tokens, n_layers=args.layers or cfg.n_layers)
    if args.router_variant or args.d_m:   # ablations run with the workload's tau
        cfg = cfg.replace(router_variant=args.router_variant, d_m=args.d_m or cfg.d_m)
    default_shape = cfg == hi.CONFIGS[args.workload] and args.tau is None and args.bypass is None
    T, d, L = cfg.n_tokens, cfg.d_model, cfg.n_layers
    decoder = bool(cfg.n_heads)
    kvdec = bool(cfg.kv_decode_of)
    if decoder and not kvdec and args.tokens:
        cfg = cfg.replace(batch=max(1, cfg.n_tokens // cfg.seq_len))
    B, S = cfg.batch, cfg.seq_len
    if args.backward and (decoder or cfg.dtype != "bf16"):
        raise SystemExit("--backward runs on the bf16 routed-stack workloads")
    if kvdec and B != T:
        raise SystemExit(f"KV decoding workload needs T = batch ({B} != {T})")
    if decoder and not kvdec and B * S != T:
        raise SystemExit(f"decoder workload needs T = batch x seq_len ({B}x{S} != {T})")
    t_gen = time.time()
    w = hi.generate_weights(cfg)
    h_np = hi.generate_h_in(cfg)
    P_np = None if decoder else hi.generate_attn_delta(cfg)
    t_gen = time.time() - t_gen
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.current_stream(dev)
    t_prefill = None
    if kvdec:
        # the cache: every sequence's S-token prefix, prefilled in chunks of the prefill
        # workload's shape (untimed)
        pcfg = hi.CONFIGS[cfg.kv_decode_of]
        stack = hero.HeroDecoder(cfg, w, hi.generate_attn_weights(cfg), max_tokens=pcfg.n_tokens)
        stack.init_cache(B, S + 1)
        hp_dev = torch.from_numpy(hi.generate_h_in(pcfg)).to(dev)
        t_prefill = time.time()
        for seq0 in range(0, B, pcfg.batch):
            nb = min(pcfg.batch, B - seq0)
            stack.prefill(hp_dev[:nb * S], tau, seq0, nb, S)
        torch.cuda.synchronize()
        t_prefill = time.time() - t_prefill
        stack.check()
        del hp_dev
        pos = torch.full((B,), S, dtype=torch.int32, device=dev)
    elif decoder:
        stack = hero.HeroDecoder(cfg, w, hi.generate_attn_weights(cfg))
    else:
        stack = hero.HeroStack(cfg, w)
    h = torch.from_numpy(h_np).to(dev)
    P = None if decoder else torch.from_numpy(P_np).to(dev)
    h_out = torch.empty((T, d), dtype=torch.float32, device=dev)
    g = torch.empty((L, T), dtype=torch.float32, device=dev)
    m = torch.empty((L, T), dtype=torch.uint8, device=dev)
    c = torch.empty((L,), dtype=torch.int32, device=dev)

    def barrier():
        if dist:
            dist.barrier()

    def max_over_ranks(x):
        if not dist:
            return x
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def run(flags, st=None):
        if kvdec:
            stack.decode(h, pos, S, tau, flags=flags, h_out=h_out, gate_out=g, mask_out=m,
                         counts_out=c, stream=st or stream)
        elif decoder:
            stack.forward(h, tau, B, S, flags=flags, h_out=h_out, gate_out=g, mask_out=m,
                          counts_out=c, stream=st or stream)
        else:
            stack(h, P, tau, flags=flags, h_out=h_out, gate_out=g, mask_out=m, counts_out=c,
                  stream=st or stream)

    def timed(fn, K, sampler=None):
        barrier()
        torch.cuda.synchronize()
        if sampler:
            sampler.start()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(K):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        clk = sampler.stop() if sampler else None
        return max_over_ranks(e0.elapsed_time(e1)), clk

    if args.backward:
        return backward_arm(args, cfg, stack, hero, h, P, tau, stream, dev, world, rank, timed,
                            ClockSampler(local_rank), t_gen)

    # ---- routed stack (the metric) ----
    rflags = hero.HERO_FLAG_NO_SPECULATE if args.no_speculate else 0
    for _ in range(args.warmup):
        run(rflags)
    torch.cuda.synchronize()
    stack.check()
    sampler = ClockSampler(local_rank)
    ms, clocks = timed(lambda: run(rflags), args.steps, sampler)   # the metric: no instrumentation
    stack.check()
    # per-kernel breakdown from a separate instrumented pass (events around every launch
    # serialise launches that otherwise overlap their predecessor's tail)
    hero.hero_get_profile(stack.model, reset=True)
    hero.hero_set_profiling(stack.model, True)
    timed(lambda: run(rflags), args.steps)
    hero.hero_set_profiling(stack.model, False)
    prof = hero.hero_get_profile(stack.model, reset=True)
    stack.check()
    ms_eager = ms / args.steps
    if args.graph:
        # the stack enqueues with no host synchronisation, so one step captures into a
        # CUDA graph whose replays remove the per-launch CPU cost
        graph = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        with torch.cuda.graph(graph, stream=cap):
            run(rflags, cap)
        stream.wait_stream(cap)
        for _ in range(args.warmup):
            graph.replay()
        torch.cuda.synchronize()
        ms, clocks = timed(graph.replay, args.steps, ClockSampler(local_rank))
        stack.check()
    counts = c.cpu().numpy().astype(np.int64)
    bypass = 1.0 - counts[cfg.n_dense:].sum() / ((L - cfg.n_dense) * T)   # routed blocks
    value = world * T * args.steps / (ms / 1e3)

    # ---- dense stack, same kernels ----
    dense = None
    if not args.no_dense:
        for _ in range(2):
            run(hero.HERO_FLAG_DENSE)
        ms_dense, _ = timed(lambda: run(hero.HERO_FLAG_DENSE), args.steps)
        dense = world * T * args.steps / (ms_dense / 1e3)
        stack.check()

    # ---- end to end through the C ABI with host buffers ----
    e2e = None
    if not args.no_e2e:
        hp = torch.from_numpy(h_np).pin_memory()
        Pp = None if decoder else torch.from_numpy(P_np).pin_memory()
        ho_ = torch.empty((T, d), dtype=torch.float32).pin_memory()
        cp = torch.empty((L,), dtype=torch.int32).pin_memory()

        pos_h = torch.full((B,), S, dtype=torch.int32).pin_memory() if kvdec else None

        def run_host():
            if kvdec:
                hero.hero_decode_step(stack.model, B, pos_h.data_ptr(), S, hp.data_ptr(), tau,
                                      hero.HERO_FLAG_HOST_IO | rflags, 0, ho_.data_ptr(), 0, 0,
                                      cp.data_ptr(), stream.cuda_stream)
            elif decoder:
                hero.hero_decoder_forward(stack.model, B, S, hp.data_ptr(), tau,
                                          hero.HERO_FLAG_HOST_IO | rflags, 0, ho_.data_ptr(), 0, 0,
                                          cp.data_ptr(), stream.cuda_stream)
            else:
                hero.hero_routed_ffn_stack(stack.model, T, hp.data_ptr(), Pp.data_ptr(), tau,
                                           hero.HERO_FLAG_HOST_IO | rflags, 0, ho_.data_ptr(), 0, 0,
                                           cp.data_ptr(), stream.cuda_stream)
        run_host()
        torch.cuda.synchronize()
        ms_e2e, _ = timed(run_host, args.steps)
        stack.check()
        e2e = {"value": world * T * args.steps / (ms_e2e / 1e3), "unit": UNIT,
               "h2d_bytes_per_step": int(hp.numel() * 4 + (0 if decoder else Pp.numel() * 2)
                                         + (B * 4 if kvdec else 0)),
               "d2h_bytes_per_step": int(ho_.numel() * 4 + cp.numel() * 4)}
        assert np.array_equal(cp.numpy(), counts), "host-IO path routed differently"

    # ---- roofline of the dominant kernel ----
    peaks, peak_src = load_peaks()
    work = algorithmic_work(cfg, counts, args.steps)
    dom = max(prof, key=lambda k: prof[k][0])
    dom_ms, dom_n = prof[dom]
    roof = None
    nbytes = algorithmic_bytes(cfg, counts, args.steps)
    if dom in work and dom_ms > 0:
        peak_tf = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
        peak_bw = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        # the bound is whichever floor is higher: FLOPs at the tensor peak or bytes at HBM
        hbm = nbytes.get(dom, 0.0) / (peak_bw * 1e9) > work[dom] / (peak_tf * 1e12)
        traffic = DOMINANT_TRAFFIC.get((cfg.name, dom)) if default_shape else None
        if hbm:
            achieved = nbytes[dom] / (dom_ms / 1e3) / 1e9
            roof = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": peak_bw,
                    "unit": "GB/s", "frac": achieved / peak_bw, "traffic": traffic,
                    "peak_source": f"{peak_src} hbm_gbs",
                    "algorithmic": "weights read once per block (bf16) plus cached keys/values"}
        else:
            achieved = work[dom] / (dom_ms / 1e3) / 1e12
            roof = {"kernel": dom, "bound": "tensor", "achieved": achieved, "peak": peak_tf,
                    "unit": "TFLOP/s", "frac": achieved / peak_tf, "traffic": traffic,
                    "peak_source": f"{peak_src} bf16_tflops_sustained (kernel timed inside a long step)"}
        roof["avg_launch_ms"] = dom_ms / max(dom_n, 1)
    ffn_ms = prof["ffn_gate_up"][0] + prof["ffn_down"][0]
    ffn_tflops = (work["ffn_gate_up"] + work["ffn_down"]) / (ffn_ms / 1e3) / 1e12 if ffn_ms else None

    # ---- CPU baseline: the oracle on a bounded sample ----
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import hero_oracle as ho
        step, rows, sample = oracle_step(ho, cfg, w, h_np, tau, args.cpu_sample, P_np)
        if kvdec:
            sample = ("the oracle has no incremental form (it recomputes a sequence's prefix); "
                      + sample)
        t0 = time.perf_counter()
        step()
        dt = time.perf_counter() - t0
        cpu = {"value": len(rows) / dt, "unit": UNIT, "cores": len(os.sched_getaffinity(0)),
               "kind": "oracle", "sample": f"{sample} ({dt:.1f} s; BLAS threads = cores)"}

    launches = int(sum(n for _, n in prof.values()))
    line = {
        "metric": metric_for(cfg), "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
        "config": {"workload": workload_desc(cfg, cfg.bypass),
                   "l2": ("inputs larger than L2 (no flush): weights stream from HBM each step"
                          + ("" if decoder else ", and so does P_j")),
                   "parallelism": f"token shards, {world} rank(s), no collective",
                   **({"cuda_graph": True, "eager_ms_per_step": ms_eager} if args.graph else {})},
        "roofline": roof,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": clocks,
        "dense_value": dense,
        "routed_vs_dense": (value / dense) if dense else None,
        "bypass": bypass,
        "ffn_counts": counts.tolist(),
        "ffn_gemm_tflops": ffn_tflops,
        "ffn_gemm_frac_of_sustained": (ffn_tflops / float(peaks.get("bf16_tflops_sustained", 1700.0)))
        if ffn_tflops else None,
        "kernel_ms_per_step": {k: v[0] / args.steps for k, v in prof.items()},
        "setup_s": {"generate": t_gen, **({"prefill_cache": t_prefill} if kvdec else {})},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    stack.close()
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    sys.exit(main() or 0)
