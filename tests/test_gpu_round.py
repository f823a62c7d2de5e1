"""GPU round parity against the oracle, batch invariance, forcing and edge cases."""
import numpy as np
import pytest
import torch

import synth
from oracle import decode as od
from oracle.model import Decoder
from tests.gpu_util import NEAR_TIE, decode_all, gpu_accept, lockstep, new_engine

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny():
    w = synth.make_weights(synth.TINY, seed=synth.WEIGHT_SEED)
    return synth.TINY, w, Decoder(synth.TINY, w)


@pytest.fixture(scope="module")
def tiny_gain():
    cfg = synth.TINY.with_(n_heads=8, n_kv_heads=4)   # GQA group 2 on the tiny decoder
    w = synth.make_weights(cfg, seed=7, gain_std=0.1)
    return cfg, w, Decoder(cfg, w)


def test_tiny_workload_lockstep(tiny):
    """Tiny decoder workload: prefix 448 visual + 64 text, K = 8, about 64 rounds."""
    cfg, w, dec = tiny
    wl = synth.WORKLOADS["tiny"]
    prompt = wl.prompts()[0]
    eng = new_engine(cfg, w, max_ctx=1024, max_K=8, max_prefill=512)
    st, stats = lockstep(eng, dec, prompt, wl.K, wl.max_new, check_logits=True)
    print(f"\ntiny lockstep: {stats}")
    assert st.done and len(st.out) == wl.max_new
    assert stats.rounds >= 30
    assert stats.max_logit_err <= 3e-2
    eng.close()


@pytest.mark.parametrize("K,n_vis,n_text", [(0, 40, 23), (1, 64, 0), (4, 0, 65), (15, 100, 27),
                                            (16, 127, 1)])
def test_tiny_gqa_gains_lockstep(tiny_gain, K, n_vis, n_text):
    """GQA group 2, non-unit norm gains, ragged prefixes around page edges, K in 0..16."""
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, n_vis, n_text, index=K)
    eng = new_engine(cfg, w, max_ctx=512, max_K=16, max_prefill=96)   # prefill in chunks
    st, stats = lockstep(eng, dec, prompt, K, 48, check_logits=True)
    print(f"\nK={K}: {stats}")
    assert st.done and len(st.out) == 48
    eng.close()


def test_gpu_self_spec_equals_gpu_ar(tiny_gain):
    """Batch-invariant kernels: the GPU's self-speculative output equals its own
    greedy AR (K = 0) output token for token (the paper's AR-equivalence, here
    exact because a row's arithmetic does not depend on the window it sits in)."""
    cfg, w, _ = tiny_gain
    eng = new_engine(cfg, w, max_ctx=1024, max_K=16, max_prefill=256)
    prompt = synth.make_prompt(cfg, 200, 50, index=11)
    slots = torch.tensor([0], dtype=torch.int32, device=eng.device)
    outs = {}
    for K in (0, 3, 8, 16):
        x0 = eng.prefill(0, prompt.vis, prompt.text, 200)
        outs[K] = [x0] + decode_all(eng, slots, K, 400)[0]
        assert len(outs[K]) == 200
    assert outs[3] == outs[0] and outs[8] == outs[0] and outs[16] == outs[0]
    eng.close()


def test_forced_acceptance_hits_schedule(tiny_gain):
    """Forcing d_1..d_L to the greedy continuation makes the verifier accept exactly L."""
    cfg, w, _ = tiny_gain
    K, max_new = 16, 300
    eng = new_engine(cfg, w, max_ctx=2048, max_K=K, max_prefill=256)
    prompt = synth.make_prompt(cfg, 300, 20, index=12)
    slots = torch.tensor([0], dtype=torch.int32, device=eng.device)
    x0 = eng.prefill(0, prompt.vis, prompt.text, max_new + K + 4)
    ref = [x0] + decode_all(eng, slots, K, 1000)[0]
    P = prompt.length
    teacher = np.full(P + len(ref) + 4, -1, np.int32)
    teacher[P:P + len(ref)] = ref
    sched = synth.accept_schedule("geometric", K, 1, 200)
    from paper_2609_26638_gb300 import gs
    t_dev = torch.from_numpy(teacher).to(eng.device)
    s_dev = torch.from_numpy(sched).to(eng.device)
    force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=teacher.shape[0],
                        L_sched=s_dev.data_ptr(), L_stride=sched.shape[1])
    x0b = eng.prefill(0, prompt.vis, prompt.text, max_new)
    assert x0b == x0
    dev = eng.device
    out_tok = torch.zeros((1, K + 2), dtype=torch.int32, device=dev)
    cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    done = torch.zeros(1, dtype=torch.int32, device=dev)
    torch.cuda.synchronize(dev)
    got = [x0]
    r = 0
    while True:
        eng.round(slots, K, out_tok, cnt, done, force=force)
        eng.stream.synchronize()
        c = int(cnt.cpu()[0])
        got.extend(out_tok.cpu().numpy()[0, :c].tolist())
        if int(done.cpu()[0]):
            break
        assert c == int(sched[0, r]) + 2, (r, c, sched[0, r])
        r += 1
    assert got == ref[:max_new]
    eng.check()
    eng.close()


def test_batch_equals_single_and_ragged_finish(tiny_gain):
    """Three sequences with different prefixes and caps decoded as one batch give
    the same tokens as each decoded alone; finished ones commit nothing more."""
    cfg, w, _ = tiny_gain
    K = 6
    eng = new_engine(cfg, w, max_batch=4, max_ctx=1024, max_K=K, max_prefill=256)
    prompts = [synth.make_prompt(cfg, nv, nt, index=20 + i)
               for i, (nv, nt) in enumerate([(63, 2), (130, 5), (10, 1)])]
    caps = [40, 17, 29]
    single = []
    for i, p in enumerate(prompts):
        x0 = eng.prefill(i, p.vis, p.text, caps[i])
        single.append([x0] + decode_all(eng, torch.tensor([i], dtype=torch.int32, device=eng.device),
                                         K, 100)[0])
    x0s = [eng.prefill(i, p.vis, p.text, caps[i]) for i, p in enumerate(prompts)]
    slots = torch.tensor([2, 0, 1], dtype=torch.int32, device=eng.device)   # any slot order
    outs = decode_all(eng, slots, K, 100)
    batch = {2: outs[0], 0: outs[1], 1: outs[2]}
    for i in range(3):
        assert [x0s[i]] + batch[i] == single[i]
        assert len(single[i]) == caps[i]
    eng.close()


def test_stop_token_truncates(tiny_gain):
    cfg, w, dec = tiny_gain
    prompt = synth.make_prompt(cfg, 50, 10, index=31)
    ar = od.ar_decode(dec, od.prefill(dec, prompt.vis, prompt.text, 512, 40))
    eos = ar[9]
    eng = new_engine(cfg, w, max_ctx=512, max_K=8, max_prefill=128, eos=eos)
    st, stats = lockstep(eng, dec, prompt, 8, 40, eos=eos)
    assert st.done and st.out[-1] == eos and eos not in st.out[:-1]
    eng.close()


def test_bad_requests_raise(tiny):
    from paper_2609_26638_gb300 import gs
    cfg, w, _ = tiny
    eng = new_engine(cfg, w, max_ctx=256, max_K=4, max_prefill=128)
    dev = eng.device
    slots = torch.tensor([0], dtype=torch.int32, device=dev)
    o = torch.zeros((1, 8), dtype=torch.int32, device=dev)
    c = torch.zeros(1, dtype=torch.int32, device=dev)
    d = torch.zeros(1, dtype=torch.int32, device=dev)
    with pytest.raises(gs.GsError) as e:
        eng.round(slots, 5, o, c, d)                         # K > max_K
    assert e.value.code == gs.GS_ERR_INVALID_ARG
    force = gs.gs_force(teacher=o.data_ptr(), teacher_stride=8, L_sched=c.data_ptr(), L_stride=1)
    with pytest.raises(gs.GsError) as e:                     # forcing is a greedy-only hook
        gs.gs_round(eng.handle, slots.data_ptr(), 1, 2, gs.GS_ACCEPT_STOCHASTIC, force,
                    o.data_ptr(), c.data_ptr(), d.data_ptr())
    assert e.value.code == gs.GS_ERR_INVALID_ARG
    with pytest.raises(gs.GsError) as e:
        gs.gs_round(eng.handle, slots.data_ptr(), 1, 2, 7, None, o.data_ptr(), c.data_ptr(),
                    d.data_ptr())
    assert e.value.code == gs.GS_ERR_INVALID_ARG
    with pytest.raises(gs.GsError) as e:
        eng.set_sampling(0.0, 1)
    assert e.value.code == gs.GS_ERR_INVALID_ARG
    p = synth.make_prompt(cfg, 200, 10)
    with pytest.raises(gs.GsError) as e:
        eng.prefill(0, p.vis, p.text, 100)                   # 210 + 100 + 6 > 256
    assert e.value.code == gs.GS_ERR_OOM
    with pytest.raises(gs.GsError):
        eng.prefill(3, p.vis[:8], p.text[:2], 4)             # slot out of range
    # an unprefilled slot is "done": a round commits nothing
    eng.round(slots, 2, o, c, d)
    eng.stream.synchronize()
    assert int(c.cpu()[0]) == 0 and int(d.cpu()[0]) == 1
    # out-of-range token id: the kernel clamps it and raises the device check
    bad = p.text[:4].copy()
    bad[1] = cfg.vocab + 5
    eng.prefill(0, None, bad, 4)
    with pytest.raises(gs.GsError) as e:
        eng.check()
    assert e.value.code == gs.GS_ERR_DEVICE_CHECK
    eng.check()                                            # cleared
    eng.close()


def test_bounded_wait_times_out_and_context_survives(tiny_gain):
    """Failure detection without a GPU fault: a probe kernel waits, through the
    bounded mbarrier wait every pipeline uses, on a barrier nothing arrives on,
    with a 20 ms limit.  The wait runs out, gs_sync_check reports
    GS_ERR_TIMEOUT (then the word is clear), and the context stays usable: the
    rounds that follow commit the same tokens as before the probe."""
    from paper_2609_26638_gb300 import gs
    cfg, w, _ = tiny_gain
    eng = new_engine(cfg, w, max_ctx=512, max_K=8, max_prefill=128)
    prompt = synth.make_prompt(cfg, 40, 12, index=17)
    slots = torch.tensor([0], dtype=torch.int32, device=eng.device)
    eng.prefill(0, prompt.vis, prompt.text, 24)
    before = decode_all(eng, slots, 8, 12)[0]
    gs.gs_wait_probe(eng.handle, 20000)
    with pytest.raises(gs.GsError) as e:
        eng.check()
    assert e.value.code == gs.GS_ERR_TIMEOUT
    eng.check()                                            # cleared
    with pytest.raises(gs.GsError) as e:
        gs.gs_wait_probe(eng.handle, 0)
    assert e.value.code == gs.GS_ERR_INVALID_ARG
    eng.prefill(0, prompt.vis, prompt.text, 24)
    after = decode_all(eng, slots, 8, 12)[0]
    assert after == before
    eng.close()


def test_round_profile_matches_round(tiny_gain):
    """gs_round_profile runs the same round as gs_round (same committed tokens
    and state) and reports one timed entry per kernel launch, in launch order:
    window, embed, per layer QKV / attention / O / gate-up / down, LM head, for
    the draft and the verify forward, then accept."""
    cfg, w, _ = tiny_gain
    eng = new_engine(cfg, w, max_ctx=1024, max_K=16, max_prefill=256)
    prompt = synth.make_prompt(cfg, 120, 30, index=3)
    dev = eng.device
    slots = torch.tensor([0], dtype=torch.int32, device=dev)
    K = 6
    bufs = [torch.zeros((1, K + 2), dtype=torch.int32, device=dev),
            torch.zeros(1, dtype=torch.int32, device=dev),
            torch.zeros(1, dtype=torch.int32, device=dev)]
    eng.prefill(0, prompt.vis, prompt.text, 100)
    ref = []
    for _ in range(3):
        eng.round(slots, K, *bufs)
        eng.stream.synchronize()
        ref.append(bufs[0].cpu().numpy()[0, :int(bufs[1].cpu()[0])].tolist())
    ref_state = eng.state(0)
    eng.prefill(0, prompt.vis, prompt.text, 100)
    got = []
    for _ in range(3):
        prof = eng.round_profile(slots, K, *bufs)
        got.append(bufs[0].cpu().numpy()[0, :int(bufs[1].cpu()[0])].tolist())
    assert got == ref
    assert eng.state(0) == ref_state
    fwd = ["embed"] + ["qkv", "attention", "o_proj", "gate_up", "down"] * cfg.n_layers + ["lm_head"]
    assert [k for k, _ in prof] == ["window"] + fwd + ["window"] + fwd + ["accept"]
    assert len(prof) == gs_launches(eng)
    assert all(ms > 0 for _, ms in prof)
    eng.check()
    eng.close()


def gs_launches(eng):
    from paper_2609_26638_gb300 import gs
    return gs.gs_round_launches(eng.handle)
