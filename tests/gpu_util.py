"""Helpers for the GPU parity tests: engine construction and the oracle-driven
lock-step comparison of rounds.

Lock-step protocol.  The oracle decodes on its own (float64); before every
round the GPU sequence holds exactly the oracle's token history (if an
earlier round diverged at a near-tie, the GPU is re-prefilled with the
oracle's history and its boundary token restored).  Per round:
  * draft rows: GPU argmax == oracle argmax, except where the oracle's top-2
    gap is below NEAR_TIE;
  * verify rows (compared when the verify inputs agree): same rule;
  * the GPU round is internally consistent: its committed run is
    [a0, d_1..d_A, a_{A+1}] of its own verify inputs and predictions, cut by
    the stop rules;
  * logits (optional): max |GPU - oracle| <= the tolerance on rows whose
    inputs agree.
No value computed by the GPU is ever fed to the oracle.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

from oracle import decode as od

NEAR_TIE = 0.1          # nats, top-2 logit gap under which a flip is allowed
LOGIT_TOL = 3e-2        # max-abs logit error, 16-bit GPU path vs float64 oracle


@dataclasses.dataclass
class LockstepStats:
    rounds: int = 0
    rows: int = 0
    near_tie_flips: int = 0
    resyncs: int = 0
    max_logit_err: float = 0.0
    logit_rows: int = 0
    oracle_gap_below_tie: int = 0


def new_engine(model, weights, *, max_batch=1, max_ctx=4096, max_K=16, max_prefill=1024,
               split_pages=0, eos=None):
    from paper_2609_26638_gb300.runtime import Engine
    return Engine(model, weights, max_batch=max_batch, max_ctx=max_ctx, max_K=max_K,
                  max_prefill=max_prefill, split_pages=split_pages, eos_token_id=eos)


def gpu_accept(vin: np.ndarray, vt: np.ndarray, K: int) -> int:
    A = 0
    while A < K and vin[1 + A] == vt[A]:
        A += 1
    return A


def lockstep(eng, dec, prompt, K: int, max_new: int, max_rounds: int = 1 << 30, slot: int = 0,
             eos: int = -1, check_logits: bool = False, logit_tol: float = LOGIT_TOL,
             oracle_state=None):
    from paper_2609_26638_gb300 import gs
    dev = eng.device
    V = dec.cfg.vocab
    W = K + 1
    stats = LockstepStats()
    cap = prompt.length + 2 * max_new + K + 8
    st = oracle_state if oracle_state is not None else od.prefill(dec, prompt.vis, prompt.text,
                                                                   cap, max_new, eos)
    x0 = eng.prefill(slot, prompt.vis, prompt.text, max_new)
    if x0 != st.x0:
        assert st.prefill_gap < NEAR_TIE, ("prefill x0 differs", x0, st.x0, st.prefill_gap)
        stats.near_tie_flips += 1
        eng.restore(slot, st.n, st.x0, 1, max_new, int(st.done))

    slots = torch.tensor([slot], dtype=torch.int32, device=dev)
    out_tok = torch.zeros((1, K + 2), dtype=torch.int32, device=dev)
    out_cnt = torch.zeros(1, dtype=torch.int32, device=dev)
    out_done = torch.zeros(1, dtype=torch.int32, device=dev)
    b_draft = torch.zeros(W, dtype=torch.int32, device=dev)
    b_vin = torch.zeros(W, dtype=torch.int32, device=dev)
    b_vt = torch.zeros(W, dtype=torch.int32, device=dev)
    dbg = gs.gs_debug()
    dbg.draft_tok, dbg.verify_in, dbg.verify_tok = b_draft.data_ptr(), b_vin.data_ptr(), b_vt.data_ptr()
    if check_logits:
        dl = torch.zeros((W, V), dtype=torch.float32, device=dev)
        vl = torch.zeros((W, V), dtype=torch.float32, device=dev)
        dbg.draft_logits, dbg.verify_logits = dl.data_ptr(), vl.data_ptr()
    torch.cuda.synchronize(dev)

    while not st.done and stats.rounds < max_rounds:
        n_before = st.n
        res = od.self_spec_round(dec, st, K)
        eng.round(slots, K, out_tok, out_cnt, out_done, dbg=dbg)
        eng.stream.synchronize()
        eng.check()
        stats.rounds += 1
        g_draft = b_draft.cpu().numpy()
        g_vin = b_vin.cpu().numpy()
        g_vt = b_vt.cpu().numpy()
        cnt = int(out_cnt.cpu()[0])
        g_out = out_tok.cpu().numpy()[0, :cnt].tolist()
        stats.rows += 2 * W
        stats.oracle_gap_below_tie += int((res.draft_gap < NEAR_TIE).sum() + (res.verify_gap < NEAR_TIE).sum())

        same_inputs = True
        want_draft = np.concatenate([[res.a0], res.d_draft])
        for i in range(W):
            if g_draft[i] != want_draft[i]:
                assert res.draft_gap[i] < NEAR_TIE, (
                    f"round {stats.rounds}: draft row {i} gpu {g_draft[i]} oracle {want_draft[i]} "
                    f"gap {res.draft_gap[i]:.4f}")
                stats.near_tie_flips += 1
                same_inputs = False
        if check_logits:
            err = float(np.max(np.abs(dl.cpu().numpy().astype(np.float64) - res.draft_logits)))
            assert err <= logit_tol, f"draft logits err {err}"
            stats.max_logit_err = max(stats.max_logit_err, err)
            stats.logit_rows += W
        if same_inputs:
            assert list(g_vin) == [res.a0] + list(res.d)
            for i in range(W):
                if g_vt[i] != res.a[i]:
                    assert res.verify_gap[i] < NEAR_TIE, (
                        f"round {stats.rounds}: verify row {i} gpu {g_vt[i]} oracle {res.a[i]} "
                        f"gap {res.verify_gap[i]:.4f}")
                    stats.near_tie_flips += 1
            if check_logits:
                err = float(np.max(np.abs(vl.cpu().numpy().astype(np.float64) - res.verify_logits)))
                assert err <= logit_tol, f"verify logits err {err}"
                stats.max_logit_err = max(stats.max_logit_err, err)
                stats.logit_rows += W
        # the GPU's own round is consistent with the acceptance rule
        A = gpu_accept(g_vin, g_vt, K)
        run = [int(g_vin[0])] + [int(x) for x in g_vin[1:1 + A]] + [int(g_vt[A])]
        assert g_out == run[:cnt] and 1 <= cnt <= A + 2
        if g_out == res.committed:
            gst = eng.state(slot)
            if not st.done:
                assert gst["seq_len"] == st.n == n_before + res.A + 2 and gst["x0"] == st.x0
        elif not st.done:
            stats.resyncs += 1
            text = np.concatenate([prompt.text, np.asarray(st.out[:-1], dtype=np.int32)])
            eng.prefill(slot, prompt.vis, text, max_new)
            eng.restore(slot, st.n, st.x0, len(st.out), max_new, int(st.done))
    return st, stats


def decode_all(eng, slots, K, max_rounds, force=None):
    """Rounds (graph launches) until every sequence in `slots` is done: per
    sequence the committed tokens after its prefill's x0."""
    dev = eng.device
    n = slots.shape[0]
    out_tok = torch.zeros((n, K + 2), dtype=torch.int32, device=dev)
    cnt = torch.zeros(n, dtype=torch.int32, device=dev)
    done = torch.zeros(n, dtype=torch.int32, device=dev)
    outs = [[] for _ in range(n)]
    torch.cuda.synchronize(dev)
    for _ in range(max_rounds):
        eng.round(slots, K, out_tok, cnt, done, force=force)
        eng.stream.synchronize()
        c = cnt.cpu().numpy()
        t = out_tok.cpu().numpy()
        for i in range(n):
            outs[i].extend(t[i, :c[i]].tolist())
        if done.cpu().numpy().all():
            break
    eng.check()
    return outs
