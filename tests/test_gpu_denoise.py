"""GPU parity of the two confidence-thresholded denoising loops against the
oracle: direct block-diffusion decoding (gs_diffusion_block) and multi-step
drafting (gs_round_refined), both one CUDA graph with a conditional loop.

A loop step's decisions (which positions a step reveals, which tokens they
take) may differ from the oracle's only where the oracle was within a
margin of flipping (oracle.decode.reveal_margin below 0.1 in log units: a
top-2 logit gap, a log-confidence distance from the threshold, or the
log-ratio of the two most confident open positions); such a block or round
is counted and the GPU sequence continues from the oracle's history.
Thresholds of -1 and 2 make the reveal pattern independent of the values
(the whole block at once; one position per step).  GPU-only properties hold
bit for bit: block size 1 is greedy AR, a batch equals each sequence alone,
tau_d < 0 is the one-shot round.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import decode as od
from oracle.model import Decoder
from tests.gpu_util import NEAR_TIE, decode_all, new_engine, oracle_teacher

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_gain():
    cfg = synth.TINY.with_(n_heads=8, n_kv_heads=4)   # GQA group 2 on the tiny decoder
    w = synth.make_weights(cfg, seed=7, gain_std=0.1)
    return cfg, w, Decoder(cfg, w)


def _bufs(dev, n, width):
    return (torch.zeros((n, width), dtype=torch.int32, device=dev),
            torch.zeros(n, dtype=torch.int32, device=dev),
            torch.zeros(n, dtype=torch.int32, device=dev),
            torch.zeros(n, dtype=torch.int32, device=dev))


def _block_margin(b: od.BlockResult, B: int, tau: float) -> float:
    m, masked = float("inf"), list(range(B))
    for step, rev in enumerate(b.revealed_per_step):
        picked = [j - 1 for j in rev]
        m = min(m, od.reveal_margin(b.conf_per_step[step], b.gap_per_step[step], masked, picked,
                                    tau))
        masked = [j for j in masked if j not in picked]
    return m


def _median_conf(dec, st, W_rows):
    logits = od.denoise_forward(dec, st.cache.copy(), st.x0, [None] * W_rows)
    return float(np.median(np.max(od.softmax_rows(logits), axis=1)))


def _resync(eng, slot, prompt, st, max_new):
    text = np.concatenate([prompt.text, np.asarray(st.out[:-1], dtype=np.int32)])
    eng.prefill(slot, prompt.vis, text, max_new)
    eng.restore(slot, st.n, st.x0, len(st.out), max_new, int(st.done))


def diffusion_lockstep(eng, dec, prompt, B, tau, max_new, max_blocks=1 << 30, st=None):
    """Blocks of the GPU against the oracle's; returns (blocks, equal, near-margin)."""
    dev = eng.device
    if st is None:
        st = od.prefill(dec, prompt.vis, prompt.text, prompt.length + 2 * max_new + 2 * B + 8,
                        max_new)
    x0 = eng.prefill(0, prompt.vis, prompt.text, max_new)
    if x0 != st.x0:
        assert st.prefill_gap < NEAR_TIE
        eng.restore(0, st.n, st.x0, 1, max_new)
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    out_tok, cnt, done, steps = _bufs(dev, 1, B)
    blocks = equal = near = 0
    while not st.done and blocks < max_blocks:
        res = od.diffusion_block(dec, st, B, tau)
        eng.diffusion_block(slots, B, tau, out_tok, cnt, done, steps)
        eng.stream.synchronize()
        blocks += 1
        got = out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist()
        g_steps = int(steps.cpu()[0])
        if got == res.committed and g_steps == res.steps:
            equal += 1
            if not st.done:
                g = eng.state(0)
                assert g["seq_len"] == st.n and g["x0"] == st.x0
            continue
        margin = _block_margin(res, B, tau)
        assert margin < NEAR_TIE, (f"block {blocks}: gpu {got} ({g_steps} steps) oracle "
                                   f"{res.committed} ({res.steps} steps), margin {margin:.4f}")
        near += 1
        if not st.done:
            _resync(eng, 0, prompt, st, max_new)
    eng.check()
    return st, blocks, equal, near


@pytest.mark.parametrize("B,tau", [(4, -1.0), (4, 2.0), (8, "median"), (16, -1.0), (5, 2.0)])
def test_diffusion_blocks_match_oracle(tiny_gain, B, tau):
    """Direct block diffusion on the tiny GQA decoder, block by block against
    the oracle (tokens, denoising steps, cache length and boundary)."""
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, 70, 26, index=B)
    max_new = 40
    st = od.prefill(dec, prompt.vis, prompt.text, prompt.length + 2 * max_new + 2 * B + 8, max_new)
    t = _median_conf(dec, st, B) if tau == "median" else tau
    eng = new_engine(cfg, w, max_ctx=512, max_K=16, max_prefill=128)
    st, blocks, equal, near = diffusion_lockstep(eng, dec, prompt, B, t, max_new, st=st)
    print(f"\nB={B} tau={t:.5f}: {blocks} blocks, {equal} equal, {near} near-margin")
    assert st.done and blocks >= (max_new - 1) // B
    assert equal + near == blocks and equal >= blocks - 2
    eng.close()


def test_diffusion_block_size_one_is_gpu_greedy_ar(tiny_gain):
    """B = 1 reveals the causal boundary row's argmax: the GPU's block diffusion
    equals its own greedy AR (K = 0 rounds) bit for bit, one step per block."""
    cfg, w, _ = tiny_gain
    prompt = synth.make_prompt(cfg, 40, 33, index=2)
    eng = new_engine(cfg, w, max_ctx=512, max_K=8, max_prefill=128)
    dev = eng.device
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    x0 = eng.prefill(0, prompt.vis, prompt.text, 30)
    ar = [x0] + decode_all(eng, slots, 0, 30)[0]
    eng.prefill(0, prompt.vis, prompt.text, 30)
    out_tok, cnt, done, steps = _bufs(dev, 1, 1)
    got = [x0]
    for _ in range(40):
        eng.diffusion_block(slots, 1, 0.5, out_tok, cnt, done, steps)
        eng.stream.synchronize()
        got.extend(out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist())
        assert int(steps.cpu()[0]) == 1
        if int(done.cpu()[0]):
            break
    assert got == ar
    eng.check()
    eng.close()


def test_diffusion_batch_equals_single(tiny_gain):
    """Three sequences (ragged prefixes) denoised together give each the blocks
    and step counts it gets alone: a sequence whose block completes early
    only idles while the others finish theirs."""
    cfg, w, _ = tiny_gain
    prompts = [synth.make_prompt(cfg, nv, nt, index=10 + i)
               for i, (nv, nt) in enumerate([(30, 5), (64, 1), (100, 27)])]
    B, tau, max_new, n_blocks = 6, 1.5e-3, 25, 4
    eng = new_engine(cfg, w, max_batch=3, max_ctx=512, max_K=8, max_prefill=128)
    dev = eng.device
    single = []
    for i, p in enumerate(prompts):
        eng.prefill(i, p.vis, p.text, max_new)
        slots = torch.tensor([i], dtype=torch.int32, device=dev)
        bufs = _bufs(dev, 1, B)
        seq = []
        for _ in range(n_blocks):
            eng.diffusion_block(slots, B, tau, *bufs)
            eng.stream.synchronize()
            seq.append((bufs[0].cpu().numpy()[0, :int(bufs[1].cpu()[0])].tolist(),
                        int(bufs[3].cpu()[0])))
        single.append(seq)
    for i, p in enumerate(prompts):
        eng.prefill(i, p.vis, p.text, max_new)
    order = [2, 0, 1]
    slots = torch.tensor(order, dtype=torch.int32, device=dev)
    bufs = _bufs(dev, 3, B)
    for k in range(n_blocks):
        eng.diffusion_block(slots, B, tau, *bufs)
        eng.stream.synchronize()
        for j, i in enumerate(order):
            got = (bufs[0].cpu().numpy()[j, :int(bufs[1].cpu()[j])].tolist(),
                   int(bufs[3].cpu()[j]))
            assert got == single[i][k], (i, k)
    eng.check()
    eng.close()


def refined_lockstep(eng, dec, prompt, K, tau, max_new, teacher=None, sched=None):
    dev = eng.device
    from paper_2609_26638_gb300 import gs
    st = od.prefill(dec, prompt.vis, prompt.text, prompt.length + 2 * max_new + 2 * K + 8, max_new)
    x0 = eng.prefill(0, prompt.vis, prompt.text, max_new)
    if x0 != st.x0:
        assert st.prefill_gap < NEAR_TIE
        eng.restore(0, st.n, st.x0, 1, max_new)
    force = None
    if teacher is not None:
        t_dev = torch.from_numpy(np.ascontiguousarray(teacher, dtype=np.int32)).to(dev)
        s_dev = torch.from_numpy(np.ascontiguousarray(sched, dtype=np.int32)).to(dev)
        force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=int(t_dev.shape[0]),
                            L_sched=s_dev.data_ptr(), L_stride=int(s_dev.shape[0]))
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    out_tok, cnt, done, steps = _bufs(dev, 1, K + 2)
    rounds = equal = near = 0
    while not st.done:
        L = None if teacher is None else int(sched[rounds])
        res, rec = od.self_spec_round_refined(dec, st, K, tau, teacher, L)
        eng.round_refined(slots, K, tau, out_tok, cnt, done, force=force, out_steps=steps)
        eng.stream.synchronize()
        rounds += 1
        got = out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist()
        if got == res.committed and int(steps.cpu()[0]) == rec.steps:
            equal += 1
            continue
        m, open_ = float("inf"), list(range(K + 1))
        for s, pick in enumerate(rec.fixed_per_step):
            m = min(m, od.reveal_margin(rec.conf_per_step[s], rec.gap_per_step[s], open_, pick, tau))
            open_ = [i for i in open_ if i not in pick]
        m = min(m, float(res.verify_gap.min()))
        assert m < NEAR_TIE, (f"round {rounds}: gpu {got} oracle {res.committed} margin {m:.4f}")
        near += 1
        if not st.done:
            text = np.concatenate([prompt.text, np.asarray(st.out[:-1], dtype=np.int32)])
            eng.prefill(0, prompt.vis, text, max_new)
            eng.restore(0, st.n, st.x0, len(st.out), max_new, 0, rounds)
    eng.check()
    return st, rounds, equal, near


@pytest.mark.parametrize("K,tau", [(6, -1.0), (6, 2.0), (8, "median"), (3, 2.0)])
def test_refined_rounds_match_oracle(tiny_gain, K, tau):
    """Multi-step drafting, round by round against the oracle (committed run
    and draft forwards); the whole output equals the oracle's greedy AR."""
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, 50, 19, index=20 + K)
    max_new = 36
    st0 = od.prefill(dec, prompt.vis, prompt.text, 512, max_new)
    t = _median_conf(dec, st0, K) if tau == "median" else tau
    ar = od.ar_decode(dec, st0)
    eng = new_engine(cfg, w, max_ctx=512, max_K=16, max_prefill=128)
    st, rounds, equal, near = refined_lockstep(eng, dec, prompt, K, t, max_new)
    print(f"\nK={K} tau_d={t:.5f}: {rounds} rounds, {equal} equal, {near} near-margin")
    assert st.out == ar and equal >= rounds - 2
    eng.close()


def test_refined_forced_rounds_match_oracle(tiny_gain):
    """Forcing applies to the refined draft: with the oracle's greedy
    continuation as the teacher, both sides accept exactly L per round."""
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, 44, 12, index=41)
    K, max_new = 6, 40
    sched = np.array([0, K, 2, 5, 1, 3, 0, K, 4, 2, 2, 2, 2, 2, 2, 2, 2, 2], np.int32)
    teacher = oracle_teacher(dec, prompt, max_new + K + 4)
    eng = new_engine(cfg, w, max_ctx=512, max_K=16, max_prefill=128)
    st, rounds, equal, near = refined_lockstep(eng, dec, prompt, K, 1e-3, max_new, teacher, sched)
    assert equal >= rounds - 1 and st.out == list(teacher[prompt.length:prompt.length + max_new])
    eng.close()


def test_refined_below_zero_is_the_one_shot_round(tiny_gain):
    """tau_d < 0 fixes every prediction after one draft forward: the round is
    gs_round's, bit for bit (same committed runs, same sequence state), and it
    reports one draft forward."""
    cfg, w, _ = tiny_gain
    prompt = synth.make_prompt(cfg, 80, 9, index=5)
    K = 7
    eng = new_engine(cfg, w, max_ctx=512, max_K=8, max_prefill=128)
    dev = eng.device
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    eng.prefill(0, prompt.vis, prompt.text, 60)
    ref = decode_all(eng, slots, K, 60)[0]
    eng.prefill(0, prompt.vis, prompt.text, 60)
    out_tok, cnt, done, steps = _bufs(dev, 1, K + 2)
    got = []
    for _ in range(60):
        eng.round_refined(slots, K, -1.0, out_tok, cnt, done, out_steps=steps)
        eng.stream.synchronize()
        got.extend(out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist())
        assert int(steps.cpu()[0]) == 1
        if int(done.cpu()[0]):
            break
    assert got == ref
    eng.check()
    eng.close()
