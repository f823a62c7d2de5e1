"""Parity at the GLM-OCR-scale decoder (24 layers, d 1024, 16 query / 8 KV
heads, SwiGLU 4096, vocab 59392) and the benchmark workloads' sizes.

The float64 oracle cannot decode whole workloads at this scale within test
time, so it checks sampled rounds and sampled sequences:
  * batch 1, prefix 2048, K = 16: lock-step rounds with logits (debug path),
    forced rounds with the oracle's own greedy continuation as the teacher
    (L = 0, L = K and values between; same teacher and schedule on both
    sides), and rounds launched exactly as the benchmark launches them
    (cached CUDA graphs, no debug outputs), committed tokens against the
    oracle's;
  * batch 32, prefixes U[1024, 6144], K = 16: the batched graph rounds of four
    sequences (the two shortest, a middle one and the longest prefix) against
    the oracle, every (sequence, round) pair compared;
  * batch 8, prefix 8192 (7168 visual), K = 32, heavy-tailed forced schedule:
    lock-step rounds with logits of one long page;
  * K = 32 on the same decoder at prefix 1024.
A committed run may differ from the oracle's only where the oracle row that
decides the first differing token has a top-2 gap below 0.1 (then the GPU
sequence is re-synchronised to the oracle's history and compared further).
Properties that hold at any size check the rest on the GPU alone: the
self-speculative output equals greedy AR (K = 0) token for token, a batch
gives each sequence the tokens it gets alone, and forcing hits the schedule,
at the full prefixes (2048, U[1024, 6144], 8192).
"""
import numpy as np
import pytest
import torch

import synth
from oracle import decode as od
from oracle.model import Decoder
from tests.gpu_util import (NEAR_TIE, decode_all, divergence_gap, lockstep, new_engine,
                            oracle_teacher, resync)

pytestmark = pytest.mark.gpu

GLM = synth.GLM


@pytest.fixture(scope="module")
def glm():
    w = synth.make_weights(GLM, seed=synth.WEIGHT_SEED)
    return w, Decoder(GLM, w)


@pytest.fixture(scope="module")
def glm_b1_state(glm):
    """The oracle's prefill of the batch-1 prompt (shared; tests take copies)."""
    _, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    return od.prefill(dec, prompt.vis, prompt.text, prompt.length + 700, wl.max_new)


def _copy_state(st):
    return od.SeqState(cache=st.cache.copy(), x0=st.x0, out=list(st.out), max_new=st.max_new,
                       eos=st.eos, done=st.done, prefill_gap=st.prefill_gap)


def _bufs(dev, n, K):
    return (torch.zeros((n, K + 2), dtype=torch.int32, device=dev),
            torch.zeros(n, dtype=torch.int32, device=dev),
            torch.zeros(n, dtype=torch.int32, device=dev))


def _graph_rounds_vs_oracle(eng, dec, seqs, slots_list, K, n_rounds, max_new):
    """Batched graph rounds over `slots_list` (as the benchmark launches them).
    `seqs` maps an index into slots_list to (prompt, oracle SeqState); each of
    those sequences runs its own oracle round every round and its committed
    run must equal the oracle's, unless the oracle row that decides the first
    differing token is a near-tie (divergence_gap < NEAR_TIE): then the GPU
    sequence is re-synchronised to the oracle's history.  Returns
    (compared pairs, near-tie divergences)."""
    dev = eng.device
    slots = torch.tensor(slots_list, dtype=torch.int32, device=dev)
    out_tok, out_cnt, out_done = _bufs(dev, len(slots_list), K)
    compared = flips = 0
    for r in range(n_rounds):
        eng.round(slots, K, out_tok, out_cnt, out_done)
        eng.stream.synchronize()
        cnt = out_cnt.cpu().numpy()
        tok = out_tok.cpu().numpy()
        for i, (prompt, st) in seqs.items():
            if st.done:
                continue
            n_before = st.n
            res = od.self_spec_round(dec, st, K)
            got = tok[i, :cnt[i]].tolist()
            compared += 1
            if got == res.committed:
                g = eng.state(slots_list[i])
                assert g["seq_len"] == n_before + res.A + 2 == st.n and g["x0"] == st.x0, (i, r)
                continue
            gap = divergence_gap(got, res)
            assert gap < NEAR_TIE, (f"seq {i} round {r}: gpu {got} oracle {res.committed} "
                                    f"deciding row gap {gap:.4f}")
            flips += 1
            resync(eng, slots_list[i], prompt, st, max_new, r + 1)
    eng.check()
    return compared, flips


def test_glm_b1_lockstep_with_logits(glm, glm_b1_state):
    """Batch 1, prefix 1600 visual + 448 text, K = 16: draft and verify rows of
    three rounds against the oracle, logits within 3e-2."""
    w, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    eng = new_engine(GLM, w, max_ctx=prompt.length + 700, max_K=16, max_prefill=2048)
    st, stats = lockstep(eng, dec, prompt, wl.K, wl.max_new, max_rounds=3, check_logits=True,
                         oracle_state=_copy_state(glm_b1_state))
    print(f"\nglm_b1 lockstep: {stats}")
    assert stats.rounds == 3 and stats.logit_rows >= 3 * 17
    assert stats.max_logit_err <= 3e-2
    eng.close()


def test_glm_b1_graph_rounds_vs_oracle(glm, glm_b1_state):
    """Rounds launched exactly as in the benchmark (cached graphs, no debug
    outputs) commit the oracle's tokens at batch 1, prefix 2048, K = 16."""
    w, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    eng = new_engine(GLM, w, max_ctx=prompt.length + 700, max_K=16, max_prefill=2048)
    st = _copy_state(glm_b1_state)
    x0 = eng.prefill(0, prompt.vis, prompt.text, wl.max_new)
    if x0 != st.x0:       # prefill boundary at a near-tie: continue from the oracle's
        assert st.prefill_gap < NEAR_TIE
        eng.restore(0, st.n, st.x0, 1, wl.max_new)
    n, flips = _graph_rounds_vs_oracle(eng, dec, {0: (prompt, st)}, [0], wl.K, 4, wl.max_new)
    print(f"\nglm_b1 graph rounds: {n} compared, {flips} near-tie divergences")
    assert n == 4
    eng.close()


def test_glm_b1_forced_rounds_vs_oracle(glm, glm_b1_state):
    """The forcing step against the oracle: the oracle's greedy-AR
    continuation is the teacher; the same teacher and schedule (L = 0, L = K
    and values between) go to gs_force and to the oracle's
    self_spec_round(..., teacher, L).  Per round the draft and verify rows
    (logits within 3e-2) and the accepted length agree, and A = L."""
    w, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    K = wl.K
    sched = np.array([0, K, 5, 1, K - 1, 9], np.int32)
    need = int(sum(int(L) + 2 for L in sched)) + K + 4
    teacher = oracle_teacher(dec, prompt, need, state=glm_b1_state)
    eng = new_engine(GLM, w, max_ctx=prompt.length + 700, max_K=K, max_prefill=2048)
    st, stats = lockstep(eng, dec, prompt, K, wl.max_new, check_logits=True,
                         oracle_state=_copy_state(glm_b1_state), teacher=teacher, schedule=sched)
    print(f"\nglm_b1 forced lockstep: {stats}")
    assert stats.rounds == len(sched) and stats.max_logit_err <= 3e-2
    for r, (L, A_or, A_gpu) in enumerate(stats.accepted):
        assert L == int(sched[r])
        if stats.near_tie_flips == 0:
            assert A_or == L and A_gpu == L, (r, L, A_or, A_gpu)
    assert sum(a is not None for _, _, a in stats.accepted) >= len(sched) - stats.near_tie_flips
    eng.close()


def test_glm_b1_forced_decode_properties(glm):
    """The benchmark's decode at full size, GPU alone: greedy AR (K = 0),
    natural self-speculative rounds (K = 16) and forced rounds all emit the
    same tokens, and every forced round commits exactly L + 2."""
    w, _ = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    K, max_new = wl.K, 160
    eng = new_engine(GLM, w, max_ctx=prompt.length + max_new + 2 * K + 64, max_K=K,
                     max_prefill=2048)
    dev = eng.device
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    # the forcing hook reads the teacher up to slot n + K + 1 of every round:
    # decode it K + 4 tokens past the cap
    x0 = eng.prefill(0, prompt.vis, prompt.text, max_new + K + 4)
    ar_long = [x0] + decode_all(eng, slots, 0, max_new + K + 4)[0]
    ar = ar_long[:max_new]
    eng.prefill(0, prompt.vis, prompt.text, max_new)
    spec = [x0] + decode_all(eng, slots, K, max_new)[0]
    assert len(ar) == max_new and spec == ar
    P = prompt.length
    teacher = np.full(P + len(ar_long) + 8, -1, np.int32)
    teacher[P:P + len(ar_long)] = ar_long
    sched = wl.schedule()
    from paper_2609_26638_gb300 import gs
    t_dev = torch.from_numpy(teacher).to(dev)
    s_dev = torch.from_numpy(np.ascontiguousarray(sched)).to(dev)
    force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=teacher.shape[0],
                        L_sched=s_dev.data_ptr(), L_stride=sched.shape[1])
    eng.prefill(0, prompt.vis, prompt.text, max_new)
    out_tok, cnt, done = _bufs(dev, 1, K)
    got, r = [x0], 0
    while True:
        eng.round(slots, K, out_tok, cnt, done, force=force)
        eng.stream.synchronize()
        c = int(cnt.cpu()[0])
        got.extend(out_tok.cpu().numpy()[0, :c].tolist())
        if int(done.cpu()[0]):
            break
        assert c == int(sched[0, r]) + 2, (r, c, sched[0, r])
        r += 1
    assert got == ar
    eng.check()
    eng.close()


def test_serve_b32_batch_vs_single_and_oracle(glm):
    """32 sequences, prefixes U[1024, 6144] (75 % visual), K = 16: batched graph
    rounds equal each sequence decoded alone (all 32), and four sequences' (the
    two shortest, a middle one, the longest) batched rounds commit the
    oracle's tokens, every (sequence, round) pair compared."""
    w, dec = glm
    wl = synth.WORKLOADS["serve_b32"]
    prompts = wl.prompts()
    K, max_new, n_rounds = wl.K, 48, 4
    cap = max(p.length for p in prompts) + 2 * max_new + 2 * K + 16
    eng = new_engine(GLM, w, max_batch=32, max_ctx=cap, max_K=K, max_prefill=2048)
    dev = eng.device
    single = []
    for i, p in enumerate(prompts):
        x0 = eng.prefill(i, p.vis, p.text, max_new)
        single.append([x0] + decode_all(eng, torch.tensor([i], dtype=torch.int32, device=dev),
                                        K, n_rounds)[0])
    x0s = [eng.prefill(i, p.vis, p.text, max_new) for i, p in enumerate(prompts)]
    order = list(range(31, -1, -1))          # any slot order
    outs = decode_all(eng, torch.tensor(order, dtype=torch.int32, device=dev), K, n_rounds)
    for j, i in enumerate(order):
        assert [x0s[i]] + outs[j] == single[i], i

    by_len = sorted(range(32), key=lambda i: prompts[i].length)
    chosen = [by_len[0], by_len[1], by_len[16], by_len[31]]
    for i, p in enumerate(prompts):
        assert eng.prefill(i, p.vis, p.text, max_new) == x0s[i]
    seqs = {}
    for j, i in enumerate(order):
        if i in chosen:
            p = prompts[i]
            st = od.prefill(dec, p.vis, p.text, p.length + 2 * max_new + 2 * K + 8, max_new)
            if st.x0 != x0s[i]:
                assert st.prefill_gap < NEAR_TIE
                eng.restore(i, st.n, st.x0, 1, max_new)
            seqs[j] = (p, st)
    n, flips = _graph_rounds_vs_oracle(eng, dec, seqs, order, K, n_rounds, max_new)
    print(f"\nserve_b32: {n} (sequence, round) pairs compared, {flips} near-tie divergences")
    assert n == len(chosen) * n_rounds
    eng.close()


def test_glm_k32_lockstep(glm):
    """The long-page block size K = 32 (33-row windows) on the same decoder,
    prefix 1024 (896 visual + 128 text): two lock-step rounds with logits."""
    w, dec = glm
    prompt = synth.make_prompt(GLM, 896, 128, index=5)
    eng = new_engine(GLM, w, max_ctx=prompt.length + 300, max_K=32, max_prefill=2048)
    st, stats = lockstep(eng, dec, prompt, 32, 128, max_rounds=2, check_logits=True)
    print(f"\nK=32 lockstep: {stats}")
    assert stats.rounds == 2 and stats.max_logit_err <= 3e-2
    eng.close()


def test_long_b8_properties(glm):
    """Batch 8, prefix 8192 (7168 visual), K = 32, GPU alone: forced rounds with
    the long-page mixture schedule (10 % L = K, 10 % L = 0, else geometric)
    commit exactly L + 2 per sequence, and the committed tokens equal greedy
    AR (K = 0) decoded in the same batch."""
    w, _ = glm
    wl = synth.WORKLOADS["long_b8"]
    prompts = wl.prompts()
    K, max_new, n_rounds = wl.K, 240, 6
    P = prompts[0].length
    eng = new_engine(GLM, w, max_batch=8, max_ctx=P + max_new + 2 * K + 16, max_K=K,
                     max_prefill=2048)
    dev = eng.device
    slots = torch.arange(8, dtype=torch.int32, device=dev)
    x0s = [eng.prefill(i, p.vis, p.text, max_new) for i, p in enumerate(prompts)]
    ar = decode_all(eng, slots, 0, max_new)
    teacher = np.full((8, P + max_new + 8), -1, np.int32)
    for i in range(8):
        seq = [x0s[i]] + ar[i]
        assert len(seq) == max_new
        teacher[i, P:P + max_new] = seq
    sched = np.ascontiguousarray(wl.schedule())
    from paper_2609_26638_gb300 import gs
    t_dev = torch.from_numpy(teacher).to(dev)
    s_dev = torch.from_numpy(sched).to(dev)
    force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=teacher.shape[1],
                        L_sched=s_dev.data_ptr(), L_stride=sched.shape[1])
    for i, p in enumerate(prompts):
        assert eng.prefill(i, p.vis, p.text, max_new) == x0s[i]
    out_tok, cnt, done = _bufs(dev, 8, K)
    got = [[x0s[i]] for i in range(8)]
    for r in range(n_rounds):
        eng.round(slots, K, out_tok, cnt, done, force=force)
        eng.stream.synchronize()
        c = cnt.cpu().numpy()
        t = out_tok.cpu().numpy()
        for i in range(8):
            # at most 1 + 6 * 34 tokens: no round reaches the 240-token cap
            assert int(c[i]) == int(sched[i, r]) + 2, (i, r, c[i], sched[i, r])
            got[i].extend(t[i, :c[i]].tolist())
    for i in range(8):
        assert got[i] == teacher[i, P:P + len(got[i])].tolist()
    eng.check()
    eng.close()


def test_long_b8_lockstep_forced(glm):
    """The long page: prefix 8192 (7168 visual + 1024 text), K = 32, the first
    three rounds of the long-page heavy-tailed forced schedule for sequence 7
    (L = 0, then L = K, then a middle value), with the oracle's greedy
    continuation as the teacher on both sides: draft and verify rows, logits
    within 3e-2, and the accepted lengths."""
    w, dec = glm
    wl = synth.WORKLOADS["long_b8"]
    seq = 7
    prompt = wl.prompts()[seq]
    K = wl.K
    sched = np.ascontiguousarray(wl.schedule()[seq, :3])
    assert sched[0] == 0 and sched[1] == K and 0 < sched[2] < K
    need = int(sum(int(L) + 2 for L in sched)) + K + 4
    cap = prompt.length + 2 * need + 2 * K + 16
    st0 = od.prefill(dec, prompt.vis, prompt.text, cap, wl.max_new)
    teacher = oracle_teacher(dec, prompt, need, state=st0)
    eng = new_engine(GLM, w, max_ctx=cap + wl.max_new, max_K=K, max_prefill=2048)
    st, stats = lockstep(eng, dec, prompt, K, wl.max_new, check_logits=True, oracle_state=st0,
                         teacher=teacher, schedule=sched)
    print(f"\nlong_b8 forced lockstep (schedule {sched.tolist()}): {stats}")
    assert stats.rounds == len(sched) and stats.max_logit_err <= 3e-2
    assert stats.logit_rows >= 2 * (K + 1) * (len(sched) - stats.near_tie_flips)
    for r, (L, A_or, A_gpu) in enumerate(stats.accepted):
        assert L == int(sched[r])
        if A_gpu is not None and stats.near_tie_flips == 0:
            assert A_gpu == A_or == L, (r, L, A_or, A_gpu)
    eng.close()


def test_glm_diffusion_blocks_vs_oracle(glm, glm_b1_state):
    """Direct block diffusion at the GLM scale (prefix 2048, B = 16): two blocks
    revealed in one step each (tau < 0), then a block revealed one position per
    step (tau = 2), each block's tokens and steps against the oracle's."""
    from tests.test_gpu_denoise import diffusion_lockstep
    w, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    eng = new_engine(GLM, w, max_ctx=prompt.length + 700, max_K=16, max_prefill=2048)
    st, blocks, equal, near = diffusion_lockstep(eng, dec, prompt, 16, -1.0, wl.max_new,
                                                 max_blocks=2, st=_copy_state(glm_b1_state))
    print(f"\nGLM diffusion tau<0: {blocks} blocks, {equal} equal, {near} near-margin")
    assert blocks == 2 and equal + near == 2
    st, blocks, equal, near = diffusion_lockstep(eng, dec, prompt, 16, 2.0, wl.max_new,
                                                 max_blocks=1, st=_copy_state(glm_b1_state))
    print(f"GLM diffusion tau=2: {blocks} blocks, {equal} equal, {near} near-margin")
    assert blocks == 1 and equal + near == 1
    eng.close()


def test_glm_stochastic_rounds_vs_oracle(glm, glm_b1_state):
    """Stochastic rounds (T = 1, the standard acceptance-rejection rule) at the
    GLM scale: sampled drafts, acceptance, the replacement or bonus sample and
    the logits of three rounds against the oracle's same Philox draws."""
    from tests.test_gpu_sampling import stochastic_lockstep
    w, dec = glm
    wl = synth.WORKLOADS["glm_b1"]
    prompt = wl.prompts()[0]
    eng = new_engine(GLM, w, max_ctx=prompt.length + 700, max_K=16, max_prefill=2048)
    st, rounds, equal, near = stochastic_lockstep(eng, dec, prompt, 16, 1.0, 2024, wl.max_new,
                                                  check_logits=True, st=_copy_state(glm_b1_state),
                                                  max_rounds=3)
    print(f"\nGLM stochastic: {rounds} rounds, {equal} equal, {near} near-margin")
    assert rounds == 3 and equal + near == 3
    eng.close()
