"""Benchmark: greedy self-speculative decoding on one GB300 per rank.

Default workload ``serve_b32``: the GLM-OCR-scale synthetic decoder (24
layers, d_model 1024, 16 query / 8 KV heads, SwiGLU 4096, vocab 59392, random
bf16 weights) serving 32 documents at once, prefixes U[1024, 6144] (75 %
visual embeddings, 64-token KV pages, ragged), block size K = 16, 512 output
tokens per sequence, accepted draft lengths forced to a seeded
censored-geometric schedule whose realized mean over the rounds run is 9.7
(within 0.1).  The same line carries the batch-1 workload ``glm_b1`` (prefix
2048 = 1600 visual + 448 text) as an extra key.  ``--workload glm_b1`` and
``--workload long_b8`` (8 x prefix 8192, K = 32, heavy-tailed acceptance) time
the other configurations as the headline; ``--K`` and ``--accept-mean``
override the block size and the forced mean (``--K 32 --accept-mean 17.4`` is
the paper's TPF-9.7 operating point).

A step is one complete decode of every sequence: the sequence states are
rolled back to the end of the prefill (the prefill itself is untimed, as in
the paper's TPF accounting) and every round of the schedule runs as one CUDA
graph (draft forward -> forcing -> verify forward -> accept/commit).  The
metric is committed tokens per second over all sequences; per-round latencies
come from CUDA events.  The 876.6 MB of weights and the KV pages every forward
streams exceed the 129 MB L2, so no flush is needed between steps.  The same
decode with K = 0 rounds (plain greedy AR, one token per forward) is timed on
the same kernels for the speed-up the method buys.

After the timed regions (one GPU, rank 0): the float64 oracle runs a bounded
sample of forced rounds of the workload's shortest sequence on the host cores
(``cpu_baseline``), and the GPU runs the same rounds with the same teacher and
schedule; ``parity`` reports the rows compared, the argmax flips at near-ties
and the largest logit error.

--impl reference times the float64 CPU oracle on this host's cores instead
(forced rounds of the workload's shortest sequence).  Multi-GPU: replicas
(one independent decode per rank, no collective on the data path).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "committed tokens/s (greedy self-speculative decode, 1 GB300 per rank)"
UNIT = "tokens/s"


def schedule_rounds(sched: np.ndarray, max_new: int) -> int:
    """Rounds a forced schedule runs until max_new tokens are committed."""
    return synth.rounds_used(sched, max_new)


# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from
# ncu captures of the kernels as committed (summaries under profiles/), with
# the algorithmic bytes of the captured launch.  A figure is used only while
# the kernel's sources hash to the value it was taken with; it is scaled to
# another launch of the same kernel by its algorithmic bytes (attention
# traffic grows with the keys read: K and V rows, once each).
_CSRC = os.path.join(ROOT, "paper_2609_26638_gb300", "csrc")
NCU_TRAFFIC = {
    "attention_b1": dict(sources=("attention.cuh", "ptx.cuh"), bytes=4990976, algorithmic=4823040,
                         sha256="c4154e97724194c54884ba6a96d4f34400276927858e81f4dd4810b09e00183e"),
    "attention_serve": dict(sources=("attention.cuh", "ptx.cuh"), bytes=233378304,
                            algorithmic=225173504,
                            sha256="f2eb4e50dce5541dd1624732eca164b8f2d58dde484e3e6a86061e1e6dbac85a"),
    "lm_head_b1": dict(sources=("gemm_tc.cuh", "gemm.cu", "ptx.cuh"), bytes=124897280,
                       algorithmic=121669768,
                       sha256="cf843ef01b07ec00b2c8f45ea0314bd187665ee6d84ddb19be137f33e3a34ecb"),
}


def ncu_traffic(key: str, algorithmic: int):
    """Measured DRAM bytes for a launch of `algorithmic` bytes, or None once
    the kernel has changed since its capture."""
    import hashlib
    e = NCU_TRAFFIC[key]
    h = hashlib.sha256()
    for f in e["sources"]:
        with open(os.path.join(_CSRC, f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest() != e["sha256"]:
        return None
    return int(round(e["bytes"] * algorithmic / e["algorithmic"]))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), "measured"
    return 6800.0, 1900.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"gs_clocks_{os.getpid()}_{gpu_index}.csv")

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}", "--format=csv,noheader",
                 "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        mhz, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                mhz.append(float(parts[1].split()[0]))
                mx = float(parts[2].split()[0])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(mhz)}


def kernel_bytes(cfg, kind: str, T: int, ctx: list) -> int | None:
    """Algorithmic HBM bytes of one launch of `kind` over T window rows.

    Each operand counted once at its storage width: fp16 weight copies, fp16
    activations, float32 residual stream (read and written), float32 per-128
    feature sums of squares (the folded RMSNorm), 8-byte argmax keys.  For
    attention, ctx[i] is sequence i's visible keys (cached prefix + window):
    K and V rows of every KV head, plus the fp16 queries read and outputs
    written.  None for the small window / accept kernels (no bandwidth model).
    """
    d, F, V = cfg.d_model, cfg.d_ffn, cfg.vocab
    Hq, Hkv, hd = cfg.n_heads, cfg.n_kv_heads, cfg.head_dim
    HD, qkv = Hq * hd, cfg.qkv_dim
    ssp = T * (d // 128) * 4
    if kind == "qkv":
        return 2 * qkv * d + 2 * T * d + ssp + 2 * T * HD + 2 * T * 2 * Hkv * hd
    if kind == "attention":
        return sum(c * Hkv * hd * 2 * 2 for c in ctx) + 2 * (2 * T * HD)
    if kind == "o_proj":
        return 2 * d * HD + 2 * T * HD + 2 * 4 * T * d + 2 * T * d + ssp
    if kind == "gate_up":
        return 2 * 2 * F * d + 2 * T * d + ssp + 2 * T * F
    if kind == "down":
        return 2 * d * F + 2 * T * F + 2 * 4 * T * d + 2 * T * d + ssp
    if kind == "lm_head":
        return 2 * V * d + 2 * T * d + ssp + 8 * T
    if kind == "embed":
        return 2 * T * d + 4 * T * d + 2 * T * d + ssp
    return None


# ---------------------------------------------------------------------- GPU arm
def gemm_flops(cfg, kind: str, T: int) -> int | None:
    """Multiply-add flops (x2) of one projection launch over T rows."""
    d, F, V, HD = cfg.d_model, cfg.d_ffn, cfg.vocab, cfg.n_heads * cfg.head_dim
    rows_k = {"qkv": (cfg.qkv_dim, d), "o_proj": (d, HD), "gate_up": (2 * F, d),
              "down": (d, F), "lm_head": (V, d)}.get(kind)
    return None if rows_k is None else 2 * T * rows_k[0] * rows_k[1]


def gpu_arm(args, rank: int, world: int):
    """The GPU arm: the headline workload's timed decode, its end-to-end
    figure, the per-kernel table and, on rank 0 of a one-GPU run, the oracle
    sample (cpu_baseline) and the parity of the GPU rounds against it; with
    the default serving workload also the batch-1 workload's figures."""
    import torch

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    K = wl.K if args.K is None else args.K
    mean = wl.accept_mean if args.accept_mean is None else args.accept_mean
    weights = synth.make_weights(wl.model)
    oracle_leg = rank == 0 and world == 1 and not args.no_cpu_baseline
    res = run_decode(args, wl, K, mean, weights, dev, world, steps=args.steps, warmup=args.warmup,
                     compare_ar=args.compare_ar, kernels=True, oracle_leg=oracle_leg)
    if args.workload == "serve_b32" and args.K is None and args.accept_mean is None \
            and args.extra_b1:
        b1 = synth.WORKLOADS["glm_b1"]
        r1 = run_decode(args, b1, b1.K, b1.accept_mean, weights, dev, world,
                        steps=max(3, args.steps // 2), warmup=args.warmup, compare_ar=False,
                        kernels=False, oracle_leg=False)
        res["glm_b1"] = r1
    return res


def run_decode(args, wl, K, mean, weights, dev, world, *, steps, warmup, compare_ar, kernels,
               oracle_leg):
    import torch
    from paper_2609_26638_gb300 import gs
    from paper_2609_26638_gb300.runtime import Engine

    cfg = wl.model
    max_new = wl.max_new
    prompts = wl.prompts()
    B = len(prompts)
    P = [p.length for p in prompts]
    extra = K + 4
    # (256 spare slots: the parity leg re-prefills a sequence with its history)
    eng = Engine(cfg, weights, max_batch=B, max_ctx=max(P) + max_new + extra + K + 2 + 320,
                 max_K=K, max_prefill=2048, device=str(dev))
    stream = eng.stream
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    out_tok = torch.zeros((B, K + 2), dtype=torch.int32, device=dev)
    out_cnt = torch.zeros(B, dtype=torch.int32, device=dev)
    out_done = torch.zeros(B, dtype=torch.int32, device=dev)

    def prefill_all(cap):
        return [eng.prefill(i, p.vis, p.text, cap) for i, p in enumerate(prompts)]

    # teacher: the greedy continuation of every sequence, from natural rounds
    x0 = prefill_all(max_new + extra)
    teacher_toks = [[x] for x in x0]
    for _ in range(max_new + extra):
        eng.round(slots, K, out_tok, out_cnt, out_done)
        stream.synchronize()
        c = out_cnt.cpu().numpy()
        t = out_tok.cpu().numpy()
        for i in range(B):
            teacher_toks[i].extend(t[i, :c[i]].tolist())
        if out_done.cpu().numpy().all():
            break
    eng.check()
    stride = max(P) + max_new + extra + K + 8
    teacher = np.full((B, stride), -1, np.int32)
    for i in range(B):
        teacher[i, P[i]:P[i] + len(teacher_toks[i])] = teacher_toks[i]
    sched_all = wl.schedule(K, mean)
    Rb = [schedule_rounds(sched_all[i], max_new) for i in range(B)]
    R = max(Rb)
    sched = np.ascontiguousarray(sched_all[:, :R + 1])
    realized = synth.realized_mean(sched_all, max_new)
    t_dev = torch.from_numpy(teacher).to(dev)
    s_dev = torch.from_numpy(sched).to(dev)
    force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=stride, L_sched=s_dev.data_ptr(),
                        L_stride=sched.shape[1])
    ring_tok = torch.zeros((R, B, K + 2), dtype=torch.int32, device=dev)
    ring_cnt = torch.zeros((R, B), dtype=torch.int32, device=dev)
    torch.cuda.synchronize(dev)

    def restore_all():
        for i in range(B):
            eng.restore(i, P[i], x0[i], 1, max_new, 0, 0)

    def one_decode(evs=None, Kr=K, frc=force, rounds=R, rt=ring_tok, rc=ring_cnt):
        restore_all()
        for r in range(rounds):
            if evs is not None:
                evs[r][0].record(stream)
            eng.round(slots, Kr, out_tok, out_cnt, out_done, force=frc)
            if evs is not None:
                evs[r][1].record(stream)
            if rt is not None:
                with torch.cuda.stream(stream):
                    rt[r].copy_(out_tok, non_blocking=True)
                    rc[r].copy_(out_cnt, non_blocking=True)

    for _ in range(warmup):
        one_decode()
    stream.synchronize()
    launches_per_round = gs.gs_round_launches(eng.handle)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize(dev)

    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(R)] for _ in range(steps)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    # GS_PROFILE_RANGE=1 marks the first timed decode as the profiler's capture
    # range (ncu --profile-from-start off); it changes no work
    prof = os.environ.get("GS_PROFILE_RANGE") == "1"
    barrier()
    with ClockSampler(dev.index) as clk:
        t0.record(stream)
        for s in range(steps):
            if prof and s == 0:
                torch.cuda.profiler.start()
            one_decode(ev[s])
            if prof and s == 0:
                stream.synchronize()
                torch.cuda.profiler.stop()
        t1.record(stream)
        stream.synchronize()
    barrier()
    elapsed = t0.elapsed_time(t1) / 1e3
    round_ms = sorted(a.elapsed_time(b) for step in ev for (a, b) in step)
    eng.check()

    # every forced round committed exactly L + 2 tokens (until the cap) and the
    # output of every sequence is its greedy continuation
    cnt = ring_cnt.cpu().numpy()
    toks = ring_tok.cpu().numpy()
    ok_sched, ok_tokens = True, True
    for i in range(B):
        got = [x0[i]]
        for r in range(R):
            got.extend(toks[r, i, :cnt[r, i]].tolist())
        ok_tokens &= got == teacher_toks[i][:max_new]
        ok_sched &= all(int(cnt[r, i]) == int(sched[i, r]) + 2 for r in range(Rb[i] - 1))
    committed_per_decode = int(cnt.sum())

    # end to end: inputs from pinned host memory, outputs back to the host, every step
    h_teacher = torch.from_numpy(teacher).pin_memory()
    h_sched = torch.from_numpy(sched).pin_memory()
    h_ring = torch.empty((R, B, K + 2), dtype=torch.int32).pin_memory()
    h_cnt = torch.empty((R, B), dtype=torch.int32).pin_memory()
    barrier()
    e0 = time.perf_counter()
    for s in range(steps):
        with torch.cuda.stream(stream):
            t_dev.copy_(h_teacher, non_blocking=True)
            s_dev.copy_(h_sched, non_blocking=True)
        one_decode()
        with torch.cuda.stream(stream):
            h_ring.copy_(ring_tok, non_blocking=True)
            h_cnt.copy_(ring_cnt, non_blocking=True)
        stream.synchronize()
    barrier()
    e_elapsed = time.perf_counter() - e0

    # plain greedy AR on the same kernels (K = 0 rounds: two one-token forwards,
    # two tokens per round), for the speed-up the method buys on this GPU
    ar = None
    if compare_ar:
        R_ar = (max_new + 1) // 2
        one_decode(Kr=0, frc=None, rounds=R_ar, rt=None)
        stream.synchronize()
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        n_ar = max(1, min(steps, 3))
        a0.record(stream)
        for _ in range(n_ar):
            one_decode(Kr=0, frc=None, rounds=R_ar, rt=None)
        a1.record(stream)
        stream.synchronize()
        eng.check()
        ar_s = a0.elapsed_time(a1) / 1e3 / n_ar
        ar = {"value": round(B * (max_new - 1) / ar_s, 1), "unit": UNIT,
              "ms_per_step": round(1e3 * ar_s, 3), "steps": n_ar, "rounds_per_step": R_ar}

    res = dict(elapsed=elapsed, e2e_elapsed=e_elapsed, tokens=committed_per_decode * steps,
               steps=steps, round_ms=round_ms, rounds=R, launches_per_round=launches_per_round,
               ok_sched=ok_sched, ok_tokens=ok_tokens, clocks=clk.summary(), ar=ar, B=B, K=K,
               mean=mean, realized_mean=round(realized, 3),
               h2d=int(teacher.nbytes + sched.nbytes),
               d2h=int(R * B * (K + 2) * 4 + R * B * 4), max_new=max_new)
    if kernels:
        res.update(kernel_table(eng, cfg, slots, K, B, R, force, out_tok, out_cnt, out_done,
                                restore_all))
        res["lm_head"] = lm_head_roofline(cfg, K, dev) if B == 1 else None
        res["attention"] = attention_roofline(cfg, dev)
    if oracle_leg:
        sample = oracle_sample(wl, 6, 1, 25.0, K, mean, weights)
        res["cpu_sample"] = sample
        res["parity"] = gpu_oracle_parity(eng, wl, sample, K)
    eng.close()
    return res


def kernel_table(eng, cfg, slots, K, B, R, force, out_tok, out_cnt, out_done, restore_all):
    """Per-kernel device times: the forced decode once more, every round
    replayed as a graph with a CUDA event after each launch (gs_round_profile);
    per kind the algorithmic bytes and flops per launch, and the roofline line
    of the kind with the largest total time."""
    hbm, bf16_tf, src = load_peaks()
    W = K + 1
    T = B * W
    per = {}
    restore_all()
    for r in range(R):
        ctx = []
        for i in range(B):
            st = eng.state(i)
            if not st["done"]:
                ctx.append(st["seq_len"] + W)
        for name, ms in eng.round_profile(slots, K, out_tok, out_cnt, out_done, force=force):
            e = per.setdefault(name, [0, 0.0, 0, 0])
            e[0] += 1
            e[1] += ms
            e[2] += kernel_bytes(cfg, name, T, ctx) or 0
            e[3] += gemm_flops(cfg, name, T) or 0
    eng.check()
    kernels = {}
    ridge = bf16_tf * 1e12 / (hbm * 1e9)
    for name, (n, ms, b, f) in sorted(per.items(), key=lambda kv: -kv[1][1]):
        k = {"launches": n, "total_ms": round(ms, 3), "us_per_launch": round(1e3 * ms / n, 2)}
        if b:
            k["bytes_per_launch"] = b // n
            k["gb_s"] = round(b / (ms * 1e-3) / 1e9, 1)
            k["frac_hbm"] = round(b / (ms * 1e-3) / 1e9 / hbm, 4)
        if f:
            k["flops_per_launch"] = f // n
            k["tflop_s"] = round(f / (ms * 1e-3) / 1e12, 1)
            k["frac_tensor"] = round(f / (ms * 1e-3) / 1e12 / bf16_tf, 4)
            k["bound"] = "tensor" if b and f / b > ridge else "hbm"
        elif b:
            k["bound"] = "hbm"
        kernels[name] = k
    dom = max((n for n in kernels if "bound" in kernels[n]), key=lambda n: kernels[n]["total_ms"])
    dk = kernels[dom]
    timing = ("CUDA event nodes after every launch of one forced decode, each round captured and "
              "replayed as a graph (no host gaps; no launch overlap across an event)")
    if dk["bound"] == "tensor":
        roof = {"kernel": f"{dom} (gemm_tc_kernel), {T} rows", "bound": "tensor",
                "achieved": dk["tflop_s"], "peak": bf16_tf, "unit": "TFLOP/s",
                "frac": dk["frac_tensor"], "peak_source": src + " bf16 burst (fp16 runs at the same rate)",
                "algorithmic_flops_per_launch": dk["flops_per_launch"],
                "us_per_launch": dk["us_per_launch"], "launches_per_step": dk["launches"],
                "timing": timing, "traffic": None}
    else:
        traffic = None
        if dom == "attention":
            traffic = ncu_traffic("attention_b1" if B == 1 else "attention_serve",
                                  dk["bytes_per_launch"])
        roof = {"kernel": f"{dom} (gemm_tc_kernel / attn_paged_kernel by kind), {T} rows",
                "bound": "hbm", "achieved": dk["gb_s"], "peak": hbm, "unit": "GB/s",
                "frac": dk["frac_hbm"], "peak_source": src,
                "algorithmic_bytes_per_launch": dk["bytes_per_launch"],
                "us_per_launch": dk["us_per_launch"], "launches_per_step": dk["launches"],
                "timing": timing, "traffic": traffic,
                "traffic_source": "ncu dram bytes of the standalone kernel, scaled by algorithmic bytes"
                if traffic is not None else None}
    gemm = {n: {"frac_tensor": kernels[n].get("frac_tensor"), "tflop_s": kernels[n].get("tflop_s"),
                "frac_hbm": kernels[n].get("frac_hbm"), "bound": kernels[n].get("bound")}
            for n in ("qkv", "o_proj", "gate_up", "down", "lm_head") if n in kernels}
    return {"roofline": roof, "kernels": kernels, "gemm_fracs": gemm}


def job_totals(elapsed: float, e2e_elapsed: float, tokens: int, world: int, device):
    """Whole-job figures over the ranks (replicas, one per GPU): the slowest
    rank's timed and end-to-end seconds (max) and the tokens every rank
    committed (sum).  One rank: the inputs."""
    if world <= 1:
        return elapsed, e2e_elapsed, tokens
    import torch
    import torch.distributed as dist
    t = torch.tensor([elapsed, e2e_elapsed], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    n = torch.tensor([float(tokens)], dtype=torch.float64, device=device)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t[0]), float(t[1]), int(round(float(n[0])))


def _time_kernel(fn, iters: int):
    """Average device seconds of one fn() launch: `iters` launches captured as
    one CUDA graph and replayed, so no host enqueue time falls between them.
    fn enqueues on torch's current stream at call time."""
    import torch
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(3):
            fn()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for _ in range(iters):
            fn()
    g.replay()
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    stream = torch.cuda.current_stream()
    a.record(stream)
    g.replay()
    b.record(stream)
    b.synchronize()
    return a.elapsed_time(b) / 1e3 / iters


def lm_head_roofline(cfg, K, dev):
    """LM-head GEMM + argmax at the decode shape (17 rows x 59392 x 1024), the
    same kernel instantiation the round launches, over rotating weight copies
    (3 x 121.6 MB > L2), 30 launches replayed as one graph."""
    import torch
    from paper_2609_26638_gb300 import gs
    hbm, _, src = load_peaks()
    M, N, Kd = K + 1, cfg.vocab, cfg.d_model
    g = torch.Generator(device=dev).manual_seed(0)
    ws = [(0.02 * torch.randn(N, Kd, device=dev, generator=g)).half() for _ in range(3)]
    x = torch.randn(M, Kd, device=dev, generator=g).half()
    keys = torch.zeros(M, dtype=torch.int64, device=dev)
    sb = gs.gs_linear_scratch_bytes(M, N, 1)
    scratch = torch.zeros(sb, dtype=torch.uint8, device=dev)
    it = [0]

    def fn():
        w = ws[it[0] % 3]
        it[0] += 1
        gs.gs_linear(x.data_ptr(), w.data_ptr(), keys.data_ptr(), M, N, Kd, gs.EPI_ARGMAX, 1,
                     scratch.data_ptr(), sb, torch.cuda.current_stream(dev).cuda_stream)

    t = _time_kernel(fn, 30)
    algo = N * Kd * 2 + M * Kd * 2 + M * 8
    achieved = algo / t / 1e9
    return {"kernel": "gemm_tc_kernel<32, argmax> (LM head 17x59392x1024)", "bound": "hbm",
            "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
            "frac": round(achieved / hbm, 4), "peak_source": src, "algorithmic_bytes": algo,
            "us_per_launch": round(t * 1e6, 2), "traffic": ncu_traffic("lm_head_b1", algo)}


def gemm_serve_rooflines(cfg, dev, T=544):
    """The four projections at the serving window (32 sequences x 17 rows) alone,
    through gs_linear with the decoder's split-K factors (so the same tile plans
    and kernels as the round), over rotating weight copies larger than L2.
    Down first (the single-kernel ncu capture takes the first launches)."""
    import torch
    from paper_2609_26638_gb300 import gs
    _, bf16_tf, src = load_peaks()
    d, F, HD = cfg.d_model, cfg.d_ffn, cfg.n_heads * cfg.head_dim
    # name, N (output features), K, epilogue, split-K as the decoder plans it
    shapes = [("down", d, F, gs.EPI_RESID_F32, 8), ("gate_up", F, d, gs.EPI_SWIGLU, 4),
              ("qkv", cfg.qkv_dim, d, gs.EPI_STORE_F16, 8), ("o_proj", d, HD, gs.EPI_RESID_F32, 8)]
    g = torch.Generator(device=dev).manual_seed(0)
    out = []
    for name, N, Kd, epi, split in shapes:
        wrows = 2 * N if epi == gs.EPI_SWIGLU else N
        n_copy = max(1, math.ceil(300e6 / (wrows * Kd * 2)))
        ws = [(0.02 * torch.randn(wrows, Kd, device=dev, generator=g)).half() for _ in range(n_copy)]
        x = torch.randn(T, Kd, device=dev, generator=g).half()
        y = torch.zeros(T, N, dtype=torch.float32 if epi == gs.EPI_RESID_F32 else torch.float16,
                        device=dev)
        sb = gs.gs_linear_scratch_bytes(T, N, split)
        scratch = torch.zeros(sb, dtype=torch.uint8, device=dev)
        it = [0]

        def fn():
            w = ws[it[0] % n_copy]
            it[0] += 1
            gs.gs_linear(x.data_ptr(), w.data_ptr(), y.data_ptr(), T, N, Kd, epi, split,
                         scratch.data_ptr(), sb, torch.cuda.current_stream(dev).cuda_stream)

        t = _time_kernel(fn, 20)
        flops = 2 * T * wrows * Kd
        tf = flops / t / 1e12
        out.append({"kernel": f"gemm_tc_kernel ({name}, {T} x {wrows} x {Kd}, split-K {split})",
                    "bound": "tensor", "achieved": round(tf, 1), "peak": bf16_tf, "unit": "TFLOP/s",
                    "frac": round(tf / bf16_tf, 4), "peak_source": src + " bf16 burst",
                    "flops": flops, "us_per_launch": round(t * 1e6, 2)})
        del ws
        torch.cuda.empty_cache()
    return out


def attention_roofline(cfg, dev, ns=None, K=16, mode=0):
    """Hybrid-mask attention alone over a paged pool (mode 0: draft masks, 1:
    verify masks).  Default shape: the serving one (32 sequences, prefix
    U[1024, 6144] -> mean ~3600, K = 16, a pool larger than L2); `ns` gives
    other cached lengths (one per sequence)."""
    import torch
    from paper_2609_26638_gb300 import gs
    hbm, _, src = load_peaks()
    rng = np.random.default_rng(5)
    if ns is None:
        ns = rng.integers(1024, 6145, size=32).astype(np.int32)
    ns = np.asarray(ns, np.int32)
    B = len(ns)
    W = K + 1
    Hq, Hkv = cfg.n_heads, cfg.n_kv_heads
    pages_per = [math.ceil((n + W + 1) / 64) for n in ns]
    pt_stride = max(pages_per)
    n_pages = sum(pages_per)
    perm = rng.permutation(n_pages)
    pt = np.full((B, pt_stride), -1, np.int32)
    o = 0
    for b in range(B):
        pt[b, :pages_per[b]] = perm[o:o + pages_per[b]]
        o += pages_per[b]
    # enough pool copies (rotated per launch) that every launch reads from DRAM
    n_copy = max(1, min(64, math.ceil(300e6 / (n_pages * 2 * Hkv * 4096 * 2))))
    kvs = [torch.randn(n_pages * 2 * Hkv * 64 * 64, device=dev).half() for _ in range(n_copy)]
    q = torch.randn(B * W * Hq * 64, device=dev).half()
    out = torch.zeros_like(q)
    ptd = torch.from_numpy(pt).to(dev)
    nd = torch.from_numpy(ns).to(dev)
    # the engine's default: at most 16 items per sequence when a batch of them
    # fits about one wave of CTAs, else at most 8
    items = 16 if B * Hkv * 16 <= 2 * 152 else 8
    sp = max(2, math.ceil(pt_stride / items))
    sb = gs.gs_attention_scratch_bytes(B, W, Hq, Hkv, pt_stride, sp)
    scratch = torch.zeros(sb, dtype=torch.uint8, device=dev)
    it = [0]

    def fn():
        kv = kvs[it[0] % n_copy]
        it[0] += 1
        gs.gs_attention(mode, q.data_ptr(), kv.data_ptr(), n_pages, ptd.data_ptr(), pt_stride,
                        nd.data_ptr(), B, W, Hq, Hkv, out.data_ptr(), scratch.data_ptr(), sb, sp,
                        torch.cuda.current_stream(dev).cuda_stream)

    t = _time_kernel(fn, 64 if B == 1 else 20)
    keys = int(sum(int(n) + W + mode for n in ns))   # the verify window reaches one slot further
    algo = keys * Hkv * 64 * 2 * 2 + 2 * B * W * Hq * 64 * 2
    achieved = algo / t / 1e9
    return {"kernel": f"attn_paged_kernel ({'verify' if mode else 'draft'}, {B} seqs, mean cached "
                      f"{int(ns.mean())}, K={K}, {sp} pages per item)", "bound": "hbm",
            "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
            "frac": round(achieved / hbm, 4), "kv_bytes": algo, "us_per_launch": round(t * 1e6, 2),
            "traffic": ncu_traffic("attention_b1" if B == 1 else "attention_serve", algo)}


# ---------------------------------------------------------------------- oracle arm
def oracle_sample(wl, n_rounds: int, warmup: int, budget_s: float, K: int, mean: float,
                  weights=None) -> dict:
    """Forced self-speculative rounds of the float64 oracle on this host's cores.

    The sample is the workload's shortest-prefix sequence (the oracle decodes
    one sequence at a time, so its tokens/s is the same for any batch): its
    own greedy AR continuation is the forcing teacher, its forced L are the
    workload's schedule for that sequence, and the timed rounds are the first
    rounds of its forced decode (prefill and teacher untimed).  Returns the
    per-round seconds and committed counts of the timed rounds, and every
    round's result with the teacher, so the GPU can run the same rounds.
    """
    from oracle import decode as od
    from oracle.model import Decoder
    cfg = wl.model
    prompts = wl.prompts()
    idx = min(range(len(prompts)), key=lambda i: prompts[i].length)
    prompt = prompts[idx]
    dec = Decoder(cfg, weights if weights is not None else synth.make_weights(cfg))
    sched = wl.schedule(K, mean)[idx]
    total = warmup + n_rounds
    need = int(sum(int(sched[r]) + 2 for r in range(total))) + K + 4
    cap = prompt.length + need + K + 8
    ar_state = od.prefill(dec, prompt.vis, prompt.text, cap, need)
    st = od.SeqState(cache=ar_state.cache.copy(), x0=ar_state.x0, out=[ar_state.x0],
                     max_new=wl.max_new, prefill_gap=ar_state.prefill_gap)
    od.ar_decode(dec, ar_state)
    P = prompt.length
    teacher = np.full(P + len(ar_state.out) + 8, -1, np.int32)
    teacher[P:P + len(ar_state.out)] = ar_state.out
    times, counts, results = [], [], []
    t_start = time.perf_counter()
    for r in range(total):
        t0 = time.perf_counter()
        res = od.self_spec_round(dec, st, K, teacher, int(sched[r]))
        dt = time.perf_counter() - t0
        results.append(res)
        if r >= warmup:
            times.append(dt)
            counts.append(len(res.committed))
            if time.perf_counter() - t_start > budget_s and len(times) >= 1:
                break
        if st.done:
            break
    return dict(times=times, counts=counts, P=P, idx=idx, results=results, teacher=teacher,
                sched=np.asarray(sched[:len(results)], np.int32), x0=st.out[0],
                prefill_gap=ar_state.prefill_gap, warmup=warmup)


NEAR_TIE = 0.1      # nats: top-2 logit gap under which an argmax flip is allowed
LOGIT_TOL = 3e-2    # max-abs logit error of the 16-bit GPU path against the float64 oracle


def gpu_oracle_parity(eng, wl, sample, K) -> dict:
    """The oracle sample's forced rounds run again on the GPU (untimed, after
    the timed region): the sequence is prefilled into its own slot, the same
    teacher and L schedule go through gs_force, and every round's draft and
    verify argmax rows, logits and committed run are compared with the
    oracle's.  An argmax may differ only where the oracle's top-2 gap is below
    0.1 (counted; the GPU sequence then continues from the oracle's history)."""
    import torch
    from paper_2609_26638_gb300 import gs
    dev = eng.device
    prompt = wl.prompts()[sample["idx"]]
    slot = sample["idx"]
    W, V = K + 1, wl.model.vocab
    max_new = wl.max_new
    out = dict(rounds=0, rows=0, logit_rows=0, near_tie_flips=0, hard_mismatches=0,
               max_logit_err=0.0, rounds_equal=0, accepted_equal=0,
               sequence=f"prefix-{sample['P']} sequence of {wl.name}, the oracle sample's "
                        f"{len(sample['results'])} forced rounds",
               near_tie=NEAR_TIE, logit_tol=LOGIT_TOL)
    x0 = eng.prefill(slot, prompt.vis, prompt.text, max_new)
    if x0 != sample["x0"]:
        out["near_tie_flips"] += 1
        out["hard_mismatches"] += int(sample["prefill_gap"] >= NEAR_TIE)
        eng.restore(slot, sample["P"], sample["x0"], 1, max_new)
    t_dev = torch.from_numpy(sample["teacher"]).to(dev)
    s_dev = torch.from_numpy(np.ascontiguousarray(sample["sched"])).to(dev)
    force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=int(t_dev.shape[0]),
                        L_sched=s_dev.data_ptr(), L_stride=int(s_dev.shape[0]))
    slots = torch.tensor([slot], dtype=torch.int32, device=dev)
    o_tok = torch.zeros((1, K + 2), dtype=torch.int32, device=dev)
    o_cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    o_done = torch.zeros(1, dtype=torch.int32, device=dev)
    b = [torch.zeros(W, dtype=torch.int32, device=dev) for _ in range(3)]
    dl = torch.zeros((W, V), dtype=torch.float32, device=dev)
    vl = torch.zeros((W, V), dtype=torch.float32, device=dev)
    dbg = gs.gs_debug(draft_tok=b[0].data_ptr(), verify_in=b[1].data_ptr(),
                      verify_tok=b[2].data_ptr(), draft_logits=dl.data_ptr(),
                      verify_logits=vl.data_ptr())
    history = [sample["x0"]]
    n = sample["P"]
    for r, res in enumerate(sample["results"]):
        eng.round(slots, K, o_tok, o_cnt, o_done, force=force, dbg=dbg)
        eng.stream.synchronize()
        g_draft, g_vin, g_vt = (x.cpu().numpy() for x in b)
        got = o_tok.cpu().numpy()[0, :int(o_cnt.cpu()[0])].tolist()
        out["rounds"] += 1
        want_draft = np.concatenate([[res.a0], res.d_draft])
        for i in range(W):
            out["rows"] += 1
            if g_draft[i] != want_draft[i]:
                out["near_tie_flips"] += 1
                out["hard_mismatches"] += int(res.draft_gap[i] >= NEAR_TIE)
        err = float(np.max(np.abs(dl.cpu().numpy().astype(np.float64) - res.draft_logits)))
        out["max_logit_err"] = max(out["max_logit_err"], err)
        out["logit_rows"] += W
        if list(g_vin) == [res.a0] + list(res.d):
            for i in range(W):
                out["rows"] += 1
                if g_vt[i] != res.a[i]:
                    out["near_tie_flips"] += 1
                    out["hard_mismatches"] += int(res.verify_gap[i] >= NEAR_TIE)
            err = float(np.max(np.abs(vl.cpu().numpy().astype(np.float64) - res.verify_logits)))
            out["max_logit_err"] = max(out["max_logit_err"], err)
            out["logit_rows"] += W
            A = 0
            while A < K and g_vin[1 + A] == g_vt[A]:
                A += 1
            out["accepted_equal"] += int(A == res.A)
        n += res.A + 2
        history.extend(res.committed)
        if got == res.committed:
            out["rounds_equal"] += 1
        else:        # continue from the oracle's history
            text = np.concatenate([prompt.text, np.asarray(history[:-1], np.int32)])
            eng.prefill(slot, prompt.vis, text, max_new)
            eng.restore(slot, n, history[-1], len(history), max_new, 0, r + 1)
    eng.check()
    out["max_logit_err"] = round(out["max_logit_err"], 5)
    return out


# ---------------------------------------------------------------------- the other decoding modes
MODE_PARAMS = {
    # stochastic acceptance (Sec. 3): temperature 1, block size K of the workload
    "stochastic": dict(temperature=1.0, seed=2024),
    # direct block diffusion (decoding appendix): block B = K, tau_c = 0.9 (the paper's sweep value)
    "diffusion": dict(tau=0.9),
    # multi-step drafting (Sec. 6): tau_d = 0.9
    "refined": dict(tau=0.9),
}
MODE_METRIC = {
    "stochastic": "committed tokens/s (stochastic self-speculative decode, T=1, 1 GB300 per rank)",
    "diffusion": "committed tokens/s (direct block-diffusion decode, tau_c=0.9, 1 GB300 per rank)",
    "refined": "committed tokens/s (multi-step drafting self-speculative decode, tau_d=0.9, "
               "1 GB300 per rank)",
}


def forward_bytes(cfg, ctx_total: int) -> int:
    """Algorithmic HBM bytes of one decoder forward over a batch whose
    sequences see ctx_total keys in all: every weight matrix once (fp16
    copies), the KV rows read once per layer (K and V, fp16)."""
    return synth.weight_bytes(cfg) + ctx_total * cfg.n_layers * cfg.n_kv_heads * cfg.head_dim * 2 * 2


def mode_arm(args, world: int):
    """One complete decode of every sequence of the workload per step in the
    given mode, each call one CUDA graph (a round, or a block with its
    conditional denoising loop).  The draws and thresholds are deterministic,
    so the calls a decode needs are counted once and then replayed without a
    host synchronisation; per call, its forwards and their context lengths
    give the algorithmic bytes of the step."""
    import torch
    from paper_2609_26638_gb300 import gs
    from paper_2609_26638_gb300.runtime import Engine
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    cfg, K, max_new, mode = wl.model, (wl.K if args.K is None else args.K), wl.max_new, args.mode
    prm = MODE_PARAMS[mode]
    prompts = wl.prompts()
    B = len(prompts)
    P = [p.length for p in prompts]
    weights = synth.make_weights(cfg)
    eng = Engine(cfg, weights, max_batch=B, max_ctx=max(P) + max_new + 2 * K + 64, max_K=K,
                 max_prefill=2048, device=str(dev))
    stream = eng.stream
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    width = K if mode == "diffusion" else K + 2
    out_tok = torch.zeros((B, width), dtype=torch.int32, device=dev)
    out_cnt = torch.zeros(B, dtype=torch.int32, device=dev)
    out_done = torch.zeros(B, dtype=torch.int32, device=dev)
    out_steps = torch.zeros(B, dtype=torch.int32, device=dev)
    x0 = [eng.prefill(i, p.vis, p.text, max_new) for i, p in enumerate(prompts)]
    if mode == "stochastic":
        eng.set_sampling(prm["temperature"], prm["seed"])

    def call():
        if mode == "stochastic":
            eng.round(slots, K, out_tok, out_cnt, out_done, rule=gs.GS_ACCEPT_STOCHASTIC)
        elif mode == "diffusion":
            eng.diffusion_block(slots, K, prm["tau"], out_tok, out_cnt, out_done, out_steps)
        else:
            eng.round_refined(slots, K, prm["tau"], out_tok, out_cnt, out_done, out_steps=out_steps)

    def restore_all():
        for i in range(B):
            eng.restore(i, P[i], x0[i], 1, max_new, 0, 0)

    # count the calls and forwards of one decode (host-synchronised, untimed)
    restore_all()
    calls, forwards, fwd_bytes, committed, launches = 0, 0, 0, 0, 0
    while True:
        ctx = [eng.state(i)["seq_len"] for i in range(B)]
        live = [not eng.state(i)["done"] for i in range(B)]
        call()
        stream.synchronize()
        calls += 1
        c = out_cnt.cpu().numpy()
        committed += int(c.sum())
        W = K + 1
        ctx_total = sum(n + W for n, lv in zip(ctx, live) if lv)
        # kernel launches of the call: a forward is embed + 5 per layer + the LM
        # head; a loop step adds its window, reveal and condition kernels
        per_fwd = 2 + 5 * cfg.n_layers
        if mode == "stochastic":
            nf = 2
            launches += 2 * per_fwd + 3                     # two windows, accept
        else:
            steps = int(out_steps.cpu().numpy().max())
            nf = steps + 1                                  # the loop's steps + verify / cache write
            launches += 1 + steps * (per_fwd + 3) + 2 + per_fwd - (1 if mode == "diffusion" else 0)
        forwards += nf
        fwd_bytes += nf * forward_bytes(cfg, ctx_total)
        if out_done.cpu().numpy().all():
            break
    eng.check()

    def one_decode():
        restore_all()
        for _ in range(calls):
            call()

    for _ in range(args.warmup):
        one_decode()
    stream.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    with ClockSampler(dev.index) as clk:
        t0.record(stream)
        for _ in range(args.steps):
            one_decode()
        t1.record(stream)
        stream.synchronize()
    elapsed = t0.elapsed_time(t1) / 1e3
    eng.check()
    # end to end: every call's committed tokens copied back to pinned host memory
    h_tok = torch.empty((B, width), dtype=torch.int32).pin_memory()
    h_cnt = torch.empty(B, dtype=torch.int32).pin_memory()
    torch.cuda.synchronize(dev)
    e0 = time.perf_counter()
    for _ in range(args.steps):
        restore_all()
        for _ in range(calls):
            call()
            with torch.cuda.stream(stream):
                h_tok.copy_(out_tok, non_blocking=True)
                h_cnt.copy_(out_cnt, non_blocking=True)
        stream.synchronize()
    e_elapsed = time.perf_counter() - e0
    eng.close()
    hbm, _, src = load_peaks()
    achieved = fwd_bytes * args.steps / elapsed / 1e9
    return dict(elapsed=elapsed, e2e_elapsed=e_elapsed, tokens=committed * args.steps, calls=calls,
                launches=launches * args.steps + args.steps * B,
                forwards=forwards, committed=committed, clocks=clk.summary(),
                roofline={"kernel": f"whole {mode} decode step (all kernels of every forward)",
                          "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm,
                          "unit": "GB/s", "frac": round(achieved / hbm, 4), "peak_source": src,
                          "algorithmic_bytes_per_step": int(fwd_bytes),
                          "traffic": None},
                d2h=int(calls * (B * width * 4 + B * 4)), B=B, K=K)


def oracle_mode_sample(wl, mode: str, K: int, budget_s: float, weights=None) -> dict:
    """The oracle in the same mode on this host's cores: the workload's
    shortest-prefix sequence from its prefill (untimed), calls timed until the
    budget is spent.  Returns committed tokens and seconds."""
    from oracle import decode as od
    from oracle import sampling as sm
    from oracle.model import Decoder
    cfg = wl.model
    prompts = wl.prompts()
    idx = min(range(len(prompts)), key=lambda i: prompts[i].length)
    prompt = prompts[idx]
    dec = Decoder(cfg, weights if weights is not None else synth.make_weights(cfg))
    st = od.prefill(dec, prompt.vis, prompt.text, prompt.length + wl.max_new + 2 * K + 8, wl.max_new)
    prm = MODE_PARAMS[mode]
    tokens, secs, calls = 0, 0.0, 0
    while not st.done and secs < budget_s:
        t0 = time.perf_counter()
        if mode == "stochastic":
            r = sm.self_spec_round_stochastic(dec, st, K, prm["temperature"], prm["seed"], idx, calls)
            n = len(r.committed)
        elif mode == "diffusion":
            n = len(od.diffusion_block(dec, st, K, prm["tau"]).committed)
        else:
            n = len(od.self_spec_round_refined(dec, st, K, prm["tau"])[0].committed)
        secs += time.perf_counter() - t0
        tokens += n
        calls += 1
    return dict(tokens=tokens, secs=secs, calls=calls, P=prompt.length)


def describe(wl, K: int, mean: float, world: int) -> dict:
    prompts = wl.prompts()
    if wl.prefix_min == wl.prefix_max:
        n_vis = int(prompts[0].vis.shape[0])
        prefix = f"prefix {wl.prefix_min} ({n_vis} visual + {wl.prefix_min - n_vis} text)"
    else:
        prefix = (f"prefixes U[{wl.prefix_min}, {wl.prefix_max}] ({round(100 * wl.vis_frac)}% visual, "
                  f"64-token pages, ragged)")
    accept = {"geometric": f"censored geometric, mean accepted length {mean} realized over the "
                           f"rounds run (within 0.1)",
              "heavy": f"10% L=K, 10% L=0, else geometric; mean accepted length {mean} realized "
                       f"over the rounds run (within 0.1)",
              "natural": f"censored geometric, mean accepted length {mean} realized over the "
                         f"rounds run (within 0.1)"}[wl.accept]
    return {"workload": f"{wl.name}: GLM-OCR-scale synthetic decoder L24 d1024 H16/8 F4096 V59392, "
                        f"batch {wl.batch}, {prefix}, K={K}, {wl.max_new} output tokens per "
                        f"sequence, forced acceptance ({accept})",
            "model": "synthetic random-init bf16 weights (seed 0)",
            "global_batch": wl.batch * max(world, 1), "K": K, "max_new": wl.max_new,
            "l2": "inputs larger than L2: 876.6 MB of weights (plus the KV pages) streamed per "
                  "forward, no flush needed",
            "parallelism": f"replicas x{max(world, 1)}"}


def decode_line(res, world: int) -> dict:
    """The figures of one timed decode (whole job over the ranks)."""
    el, ee, tokens_all = job_totals(res["elapsed"], res["e2e_elapsed"], res["tokens"], world, "cuda")
    value = tokens_all / el
    rms = res["round_ms"]
    B, steps, R = res["B"], res["steps"], res["rounds"]
    d = {"value": round(value, 1), "ms_per_step": round(1e3 * el / steps, 3),
         "round_p50_ms": round(rms[len(rms) // 2], 4),
         "round_p90_ms": round(rms[int(len(rms) * 0.9)], 4),
         "rounds_per_step": R,
         "accept_mean_realized": res["realized_mean"],
         "committed_per_round_per_seq": round(res["tokens"] / (steps * R * B), 3),
         "tpf": round(res["tokens"] / (steps * R * 2 * B), 3),
         "forced_schedule_hit": res["ok_sched"], "tokens_match_greedy": res["ok_tokens"],
         "gpu_launches": res["launches_per_round"] * R * steps + steps * B,
         "e2e": {"value": round(tokens_all / ee, 1), "unit": UNIT,
                 "h2d_bytes_per_step": res["h2d"], "d2h_bytes_per_step": res["d2h"]}}
    if res["ar"] is not None:
        d["greedy_ar"] = res["ar"]
        d["speedup_vs_greedy_ar"] = round(value / (res["ar"]["value"] * max(world, 1)), 3)
    return d


def mode_main(args, wl, world: int, rank: int) -> None:
    """The bench line of a decoding mode other than the forced greedy decode."""
    K = wl.K if args.K is None else args.K
    config = describe(wl, K, wl.accept_mean, world)
    prm = MODE_PARAMS[args.mode]
    config["workload"] = (f"{wl.name} ({args.mode} mode, {prm}): GLM-OCR-scale synthetic decoder, "
                          f"batch {wl.batch}, K (or block size) {K}, {wl.max_new} output tokens per "
                          f"sequence, natural drafting (no forcing)")
    config["mode"] = args.mode
    if args.impl == "reference":
        if rank != 0:
            return
        smp = oracle_mode_sample(wl, args.mode, K, 120.0)
        value = smp["tokens"] / smp["secs"]
        cpu = {"value": round(value, 3), "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"{smp['calls']} {args.mode} calls of the prefix-{smp['P']} sequence, float64 "
                         f"oracle on all host cores"}
        print(json.dumps({"impl": "reference", "metric": MODE_METRIC[args.mode],
                          "value": round(value, 3), "unit": UNIT, "n_gpus": args.gpus, "steps": smp["calls"],
                          "warmup": 0, "ms_per_step": round(1e3 * smp["secs"] / max(1, smp["calls"]), 2),
                          "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                          "dtype": "f64", "data": "synthetic", "config": config, "cpu_baseline": cpu,
                          "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                                  "d2h_bytes_per_step": 0}}))
        return
    import torch
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", int(os.environ["LOCAL_RANK"])))
    res = mode_arm(args, world)
    el, ee, tokens_all = job_totals(res["elapsed"], res["e2e_elapsed"], res["tokens"], world, "cuda")
    line = {"metric": MODE_METRIC[args.mode], "value": round(tokens_all / el, 1), "unit": UNIT,
            "n_gpus": max(world, 1), "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * el / args.steps, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "config": config, "calls_per_step": res["calls"], "forwards_per_step": res["forwards"],
            "tokens_per_forward": round(res["committed"] / (res["forwards"] * res["B"]), 3),
            "gpu_launches": res["launches"],
            "e2e": {"value": round(tokens_all / ee, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": res["d2h"]},
            "clocks": res["clocks"], "roofline": res["roofline"]}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        smp = oracle_mode_sample(wl, args.mode, res["K"], 25.0)
        line["cpu_baseline"] = {
            "value": round(smp["tokens"] / smp["secs"], 3), "unit": UNIT, "cores": os.cpu_count(),
            "kind": "oracle", "sample": f"{smp['calls']} {args.mode} calls of the prefix-{smp['P']} "
                                        f"sequence of the same workload, float64 oracle"}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    ap.add_argument("--workload", default="serve_b32", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--K", type=int, default=None, help="block size (default: the workload's)")
    ap.add_argument("--accept-mean", type=float, default=None,
                    help="mean forced accepted length (default: the workload's)")
    ap.add_argument("--no-compare-ar", dest="compare_ar", action="store_false",
                    help="skip timing plain greedy AR (K = 0 rounds) on the same workload")
    ap.add_argument("--no-extra-b1", dest="extra_b1", action="store_false",
                    help="with the serving workload, skip the batch-1 workload's extra figures")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mode", default="greedy", choices=["greedy", "stochastic", "diffusion", "refined"],
                    help="greedy: the forced self-speculative decode (the headline); stochastic: "
                         "GS_ACCEPT_STOCHASTIC rounds at T = 1; diffusion: direct block-diffusion "
                         "decoding, B = K, tau_c = 0.9; refined: multi-step drafting, tau_d = 0.9")
    ap.add_argument("--max-new", type=int, default=None,
                    help="output tokens per sequence (default: the workload's)")
    ap.add_argument("--kernel", default=None,
                    choices=["attention", "lm_head", "attention-sweep", "gemm-serve"],
                    help="time one kernel alone and print its roofline line (the single-kernel "
                         "ncu captures run this): attention at the workload's decode shape "
                         "(the serving batch for serve_b32), the LM head at 17 rows; "
                         "attention-sweep: one line per point of K {4,8,16,32,64} x batch "
                         "{1,8,64} x prefix {1024,4096,8192}, draft and verify masks; "
                         "gemm-serve: the four projections at the 544-row serving window")
    args = ap.parse_args()
    if args.kernel is not None:
        import torch
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        cfg = synth.WORKLOADS[args.workload].model
        K = synth.WORKLOADS[args.workload].K if args.K is None else args.K
        wl = synth.WORKLOADS[args.workload]
        if args.kernel == "gemm-serve":
            for r in gemm_serve_rooflines(cfg, dev):
                print(json.dumps(r), flush=True)
            return
        if args.kernel == "attention-sweep":
            for mode in (0, 1):
                for Ks in (4, 8, 16, 32, 64):
                    for Bs in (1, 8, 64):
                        for pre in (1024, 4096, 8192):
                            r = attention_roofline(cfg, dev, [pre] * Bs, Ks, mode)
                            r.update(mode="verify" if mode else "draft", K=Ks, batch=Bs, prefix=pre)
                            print(json.dumps(r), flush=True)
                            torch.cuda.empty_cache()
            return
        if args.kernel == "lm_head":
            r = lm_head_roofline(cfg, K, dev)
        elif wl.batch == 1:   # mid-decode of the single-sequence workload
            r = attention_roofline(cfg, dev, [wl.prefix_min + wl.max_new // 2], K)
        else:
            r = attention_roofline(cfg, dev)
        print(json.dumps(r))
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.max_new is not None:
        import dataclasses
        synth.WORKLOADS[args.workload] = dataclasses.replace(synth.WORKLOADS[args.workload],
                                                             max_new=args.max_new)
    wl = synth.WORKLOADS[args.workload]
    if args.mode != "greedy":
        mode_main(args, wl, world, rank)
        return
    K = wl.K if args.K is None else args.K
    mean = wl.accept_mean if args.accept_mean is None else args.accept_mean
    config = describe(wl, K, mean, world)

    if args.impl == "reference":
        if rank != 0:
            return
        t0 = time.perf_counter()
        smp = oracle_sample(wl, args.steps, args.warmup, 240.0, K, mean)
        times, counts = smp["times"], smp["counts"]
        value = sum(counts) / sum(times)
        cores = os.cpu_count()
        sample = (f"{len(times)} forced rounds (after {args.warmup} warm-up rounds) of the "
                  f"prefix-{smp['P']} sequence of {wl.name}, float64 oracle on all host cores "
                  f"(numpy/OpenBLAS), prefill and teacher untimed")
        line = {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
                "n_gpus": args.gpus, "steps": len(times), "warmup": args.warmup,
                "ms_per_step": round(1e3 * statistics.mean(times), 2), "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": config,
                "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": cores,
                                 "kind": "oracle", "sample": sample},
                "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0},
                "wall_s": round(time.perf_counter() - t0, 1)}
        print(json.dumps(line))
        return

    import torch
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", int(os.environ["LOCAL_RANK"])))
    res = gpu_arm(args, rank, world)
    head = decode_line(res, world)
    line = {"metric": METRIC, "value": head.pop("value"), "unit": UNIT, "n_gpus": max(world, 1),
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": head.pop("ms_per_step"), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "config": config}
    line.update(head)
    line.update({"clocks": res["clocks"], "roofline": res["roofline"],
                 "gemm_fracs": res["gemm_fracs"], "kernels": res["kernels"],
                 "attention_roofline": res["attention"]})
    if res.get("lm_head") is not None:
        line["lm_head_alone"] = res["lm_head"]
    if "glm_b1" in res:
        b1 = synth.WORKLOADS["glm_b1"]
        extra = decode_line(res["glm_b1"], world)
        extra["config"] = describe(b1, b1.K, b1.accept_mean, world)["workload"]
        extra["steps"] = res["glm_b1"]["steps"]
        line["glm_b1"] = extra
    if "parity" in res:
        line["parity"] = res["parity"]
    if "cpu_sample" in res:
        smp = res["cpu_sample"]
        line["cpu_baseline"] = {
            "value": round(sum(smp["counts"]) / sum(smp["times"]), 3), "unit": UNIT,
            "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{len(smp['times'])} forced rounds (after {smp['warmup']} warm-up) of the "
                      f"prefix-{smp['P']} sequence of the same workload, float64 oracle with "
                      f"numpy/OpenBLAS threads on all host cores"}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
