"""GPU parity of stochastic self-speculative rounds (GS_ACCEPT_STOCHASTIC)
against the oracle (oracle/sampling.py), which is pinned to the exact target
distribution on CPU.

Both sides draw the same Philox4x32-10 numbers (same seed, slot, round,
stream, row and vocabulary entry), so the sampled drafts, the acceptance
decisions and the replacement or bonus token must agree, except where the
oracle was within a margin of flipping (below 0.1 in log units): a draft
sample's Gumbel-score gap, |log r_j - log(P_j(d_j) / q_j(d_j))| of an
acceptance decision, or the replacement sample's score gap.  Such rounds
are counted and the GPU sequence continues from the oracle's history (its
round counter restored, so the streams stay aligned).  GPU-only: at
temperature -> 0 a stochastic round is the greedy round, and a batch gives
each sequence (same slot) the tokens it gets alone.
"""
import math

import numpy as np
import pytest
import torch

import synth
from oracle import decode as od
from oracle import sampling as sm
from oracle.model import Decoder
from tests.gpu_util import LOGIT_TOL, NEAR_TIE, decode_all, new_engine

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_gain():
    cfg = synth.TINY.with_(n_heads=8, n_kv_heads=4)
    w = synth.make_weights(cfg, seed=7, gain_std=0.1)
    return cfg, w, Decoder(cfg, w)


def _round_margin(res: sm.StochasticRound) -> float:
    m = float(np.min(res.draft_margin))
    for j in range(min(res.A + 1, len(res.r))):          # the decisions that were taken
        m = min(m, abs(math.log(res.r[j]) - math.log(res.accept_ratio[j])))
    return min(m, res.sample_margin)


def stochastic_lockstep(eng, dec, prompt, K, T, seed, max_new, slot=0, check_logits=False,
                        st=None, max_rounds=1 << 30):
    from paper_2609_26638_gb300 import gs
    dev = eng.device
    V = dec.cfg.vocab
    W = K + 1
    if st is None:
        st = od.prefill(dec, prompt.vis, prompt.text, prompt.length + 2 * max_new + 2 * K + 8,
                        max_new)
    x0 = eng.prefill(slot, prompt.vis, prompt.text, max_new)
    if x0 != st.x0:
        assert st.prefill_gap < NEAR_TIE
        eng.restore(slot, st.n, st.x0, 1, max_new)
    eng.set_sampling(T, seed)
    slots = torch.tensor([slot], dtype=torch.int32, device=dev)
    out_tok = torch.zeros((1, K + 2), dtype=torch.int32, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    done = torch.zeros(1, dtype=torch.int32, device=dev)
    b_draft = torch.zeros(W, dtype=torch.int32, device=dev)
    dbg = gs.gs_debug(draft_tok=b_draft.data_ptr())
    if check_logits:
        dl = torch.zeros((W, V), dtype=torch.float32, device=dev)
        vl = torch.zeros((W, V), dtype=torch.float32, device=dev)
        dbg.draft_logits, dbg.verify_logits = dl.data_ptr(), vl.data_ptr()
    rounds = equal = near = 0
    max_err = 0.0
    while not st.done and rounds < max_rounds:
        res = sm.self_spec_round_stochastic(dec, st, K, T, seed, slot, rounds)
        eng.round(slots, K, out_tok, cnt, done, dbg=dbg, rule=gs.GS_ACCEPT_STOCHASTIC)
        eng.stream.synchronize()
        rounds += 1
        got = out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist()
        draft = b_draft.cpu().numpy().tolist()
        if check_logits:
            max_err = max(max_err, float(np.max(np.abs(dl.cpu().numpy() - res.draft_logits))))
            if draft == [res.a0] + list(res.d):
                max_err = max(max_err, float(np.max(np.abs(vl.cpu().numpy() - res.verify_logits))))
        if got == res.committed and draft == [res.a0] + list(res.d):
            equal += 1
            if not st.done:
                g = eng.state(slot)
                assert g["seq_len"] == st.n and g["x0"] == st.x0 and g["rounds"] == rounds
            continue
        m = _round_margin(res)
        assert m < NEAR_TIE, (f"round {rounds}: gpu {got} draft {draft}; oracle {res.committed} "
                              f"draft {[res.a0] + list(res.d)}; margin {m:.4f}")
        near += 1
        if not st.done:
            text = np.concatenate([prompt.text, np.asarray(st.out[:-1], dtype=np.int32)])
            eng.prefill(slot, prompt.vis, text, max_new)
            eng.restore(slot, st.n, st.x0, len(st.out), max_new, 0, rounds)
    eng.check()
    assert max_err <= LOGIT_TOL
    return st, rounds, equal, near


@pytest.mark.parametrize("K,T,seed", [(6, 1.0, 1), (4, 0.7, 2), (16, 1.3, 3), (0, 1.0, 4)])
def test_stochastic_rounds_match_oracle(tiny_gain, K, T, seed):
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, 60, 21, index=50 + K)
    eng = new_engine(cfg, w, max_ctx=512, max_K=16, max_prefill=128)
    st, rounds, equal, near = stochastic_lockstep(eng, dec, prompt, K, T, seed, 40,
                                                  check_logits=True)
    print(f"\nK={K} T={T}: {rounds} rounds, {equal} equal, {near} near-margin")
    assert st.done and equal >= rounds - 2
    eng.close()


def test_zero_temperature_is_the_greedy_round(tiny_gain):
    """T -> 0: samples become argmaxes and the distributions one-hot, so the
    stochastic rounds commit the greedy rounds' tokens on the same kernels."""
    from paper_2609_26638_gb300 import gs
    cfg, w, _ = tiny_gain
    prompt = synth.make_prompt(cfg, 90, 15, index=61)
    K = 6
    eng = new_engine(cfg, w, max_ctx=512, max_K=8, max_prefill=128)
    dev = eng.device
    slots = torch.zeros(1, dtype=torch.int32, device=dev)
    eng.prefill(0, prompt.vis, prompt.text, 40)
    greedy = decode_all(eng, slots, K, 40)[0]
    eng.prefill(0, prompt.vis, prompt.text, 40)
    eng.set_sampling(1e-7, 5)
    out_tok = torch.zeros((1, K + 2), dtype=torch.int32, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    done = torch.zeros(1, dtype=torch.int32, device=dev)
    got = []
    for _ in range(40):
        eng.round(slots, K, out_tok, cnt, done, rule=gs.GS_ACCEPT_STOCHASTIC)
        eng.stream.synchronize()
        got.extend(out_tok.cpu().numpy()[0, :int(cnt.cpu()[0])].tolist())
        if int(done.cpu()[0]):
            break
    assert got == greedy
    eng.check()
    eng.close()


def test_stochastic_batch_equals_single(tiny_gain):
    """A sequence's draws depend on its slot and round count only, and every
    kernel computes a row independently of the others: batched stochastic
    rounds give each sequence the tokens it gets alone in the same slot."""
    from paper_2609_26638_gb300 import gs
    cfg, w, _ = tiny_gain
    prompts = [synth.make_prompt(cfg, nv, nt, index=70 + i)
               for i, (nv, nt) in enumerate([(20, 3), (64, 0), (90, 40)])]
    K, max_new, n_rounds = 5, 30, 5
    eng = new_engine(cfg, w, max_batch=3, max_ctx=512, max_K=8, max_prefill=128)
    eng.set_sampling(0.9, 11)
    dev = eng.device
    out_tok = torch.zeros((3, K + 2), dtype=torch.int32, device=dev)
    cnt = torch.zeros(3, dtype=torch.int32, device=dev)
    done = torch.zeros(3, dtype=torch.int32, device=dev)
    single = []
    for i, p in enumerate(prompts):
        eng.prefill(i, p.vis, p.text, max_new)
        sl = torch.tensor([i], dtype=torch.int32, device=dev)
        seq = []
        for _ in range(n_rounds):
            eng.round(sl, K, out_tok[:1], cnt[:1], done[:1], rule=gs.GS_ACCEPT_STOCHASTIC)
            eng.stream.synchronize()
            seq.append(out_tok[0, :int(cnt[0])].tolist())
        single.append(seq)
    for i, p in enumerate(prompts):
        eng.prefill(i, p.vis, p.text, max_new)
    order = [1, 2, 0]
    sl = torch.tensor(order, dtype=torch.int32, device=dev)
    for r in range(n_rounds):
        eng.round(sl, K, out_tok, cnt, done, rule=gs.GS_ACCEPT_STOCHASTIC)
        eng.stream.synchronize()
        for j, i in enumerate(order):
            assert out_tok[j, :int(cnt[j])].tolist() == single[i][r], (i, r)
    eng.check()
    eng.close()
