"""Host logic of bench.py (no GPU): the decode length of a forced schedule,
the algorithmic-byte model the roofline lines use, and the gating of the
measured DRAM traffic on the kernels' sources."""
import json
import math

import numpy as np

import bench
import synth

GLM = synth.WORKLOADS["glm_b1"].model


def test_schedule_rounds_counts_committed_tokens():
    # every round commits L + 2 tokens; the boundary token x0 is the first output
    K, max_new = 16, 512
    full = np.full(100, K, np.int64)
    assert bench.schedule_rounds(full, max_new) == math.ceil((max_new - 1) / (K + 2))
    zero = np.zeros(400, np.int64)
    assert bench.schedule_rounds(zero, max_new) == math.ceil((max_new - 1) / 2)
    sched = np.array([3, 0, 16, 5] * 50)
    n, r = 1, 0
    while n < max_new:           # brute force
        n += int(sched[r]) + 2
        r += 1
    assert bench.schedule_rounds(sched, max_new) == r


def test_weight_bytes_per_forward_match_the_model():
    # the five projection kinds at any T stream each weight once: summed over
    # the layers and the LM head they must give the model's matrix bytes
    T = 17
    per_layer = sum(bench.gemm_flops(GLM, k, T) // (2 * T) for k in ("qkv", "o_proj", "gate_up", "down"))
    total = GLM.n_layers * per_layer + bench.gemm_flops(GLM, "lm_head", T) // (2 * T)
    assert total * 2 == 876_609_536            # 438.3M fp16 weights = 876.6 MB per forward
    for kind in ("qkv", "o_proj", "gate_up", "down", "lm_head"):
        b = bench.kernel_bytes(GLM, kind, T, [])
        w = bench.gemm_flops(GLM, kind, T) // (2 * T) * 2
        assert w < b < w + 64 * T * GLM.d_ffn, kind   # weights plus per-row activation traffic


def test_attention_bytes_count_k_and_v_rows_once():
    T = 17
    ctx = [2048 + T, 3000 + T]
    b = bench.kernel_bytes(GLM, "attention", 2 * T, ctx)
    kv = sum(ctx) * GLM.n_kv_heads * GLM.head_dim * 2 * 2       # K and V, fp16
    qo = 2 * (2 * 2 * T * GLM.n_heads * GLM.head_dim)          # q read + out written, fp16
    assert b == kv + qo


def test_measured_traffic_is_gated_on_the_kernel_sources(monkeypatch):
    import hashlib
    import os
    srcs = ("gemm_tc.cuh", "gemm.cu", "ptx.cuh")
    h = hashlib.sha256()
    for f in srcs:
        with open(os.path.join(bench._CSRC, f), "rb") as fh:
            h.update(fh.read())
    cur = dict(sources=srcs, bytes=1000, algorithmic=800, sha256=h.hexdigest())
    table = dict(bench.NCU_TRAFFIC, probe=cur, stale=dict(cur, sha256="0" * 64))
    monkeypatch.setattr(bench, "NCU_TRAFFIC", table)
    assert bench.ncu_traffic("probe", 800) == 1000            # sources as captured
    assert bench.ncu_traffic("probe", 1600) == 2000           # scaled by algorithmic bytes
    assert bench.ncu_traffic("stale", 800) is None            # the kernel changed since


def test_config_names_the_workload():
    wl = synth.WORKLOADS["serve_b32"]
    d = bench.describe(wl, wl.K, wl.accept_mean, 1)
    json.dumps(d)
    assert "serve_b32" in d["workload"] and d["global_batch"] == 32 and d["K"] == wl.K
    assert bench.describe(wl, wl.K, wl.accept_mean, 4)["global_batch"] == 128


def test_mode_oracle_sample_commits_tokens():
    """The oracle leg of the other decoding modes runs on the small workload
    and reports committed tokens, calls and the sequence it sampled."""
    wl = synth.WORKLOADS["tiny"]
    for mode in ("stochastic", "diffusion", "refined"):
        smp = bench.oracle_mode_sample(wl, mode, 4, 0.5)
        assert smp["calls"] >= 1 and smp["tokens"] >= smp["calls"] and smp["secs"] > 0
        assert smp["P"] == min(p.length for p in wl.prompts())
        assert bench.MODE_METRIC[mode].startswith("committed tokens/s")


def test_forward_bytes_grow_with_context():
    """One forward reads every weight once and each sequence's cached K and V."""
    a, b = bench.forward_bytes(GLM, 0), bench.forward_bytes(GLM, 1000)
    per_key = GLM.n_layers * GLM.n_kv_heads * GLM.head_dim * 2 * 2
    assert a > 0 and b - a == 1000 * per_key
