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
    # per round: (forced L or None, oracle A, GPU A or None when the verify
    # inputs differed after a near-tie draft flip)
    accepted: list = dataclasses.field(default_factory=list)


def oracle_teacher(dec, prompt, n_tokens: int, state=None) -> np.ndarray:
    """The oracle's own greedy-AR continuation as a forcing teacher:
    teacher[p] = greedy token at absolute slot p (teacher[P] is the prefill's
    boundary token), -1 before the prefix end."""
    P = prompt.length
    cap = P + n_tokens + 8
    if state is None:
        st = od.prefill(dec, prompt.vis, prompt.text, cap, n_tokens)
    else:
        st = od.SeqState(cache=state.cache.copy(), x0=state.x0, out=[state.x0],
                         max_new=n_tokens, eos=-1)
        st.done = n_tokens <= 1
    out = od.ar_decode(dec, st)
    teacher = np.full(P + len(out) + 8, -1, np.int32)
    teacher[P:P + len(out)] = out
    return teacher


def divergence_gap(got, res) -> float:
    """Top-2 gap of the oracle row whose argmax decides the first place where
    the GPU's committed run `got` and the oracle's differ.  Every committed
    token is a verifier prediction: position 0 is a0 (draft row 0), position
    j >= 1 is a_j (verify row j-1, whose inputs are the agreeing committed
    tokens before it).  If one run is a prefix of the other, the shorter side
    rejected the next draft: that draft row (same index as its position)
    decided it.  Returns inf when the runs agree."""
    want = res.committed
    m = min(len(got), len(want))
    for j in range(m):
        if got[j] != want[j]:
            return float(res.draft_gap[0]) if j == 0 else float(res.verify_gap[j - 1])
    if len(got) == len(want):
        return float("inf")
    return float(res.draft_gap[m - 1]) if m - 1 < len(res.draft_gap) else 0.0


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
             oracle_state=None, teacher=None, schedule=None):
    """Oracle-driven lock-step (module docstring).  With `teacher` (absolute
    slot -> greedy token, from oracle_teacher) and `schedule` (forced L per
    round), both sides force the same drafts: the oracle through
    self_spec_round(..., teacher, L), the GPU through gs_force with the same
    arrays; per round the GPU's A must equal the oracle's whenever the verify
    rows agree."""
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
    force = None
    if teacher is not None:
        t_dev = torch.from_numpy(np.ascontiguousarray(teacher, dtype=np.int32)).to(dev)
        s_dev = torch.from_numpy(np.ascontiguousarray(schedule, dtype=np.int32)).to(dev)
        force = gs.gs_force(teacher=t_dev.data_ptr(), teacher_stride=int(t_dev.shape[0]),
                            L_sched=s_dev.data_ptr(), L_stride=int(s_dev.shape[0]))
        max_rounds = min(max_rounds, len(schedule))
    torch.cuda.synchronize(dev)

    while not st.done and stats.rounds < max_rounds:
        n_before = st.n
        L = None if teacher is None else int(schedule[stats.rounds])
        res = od.self_spec_round(dec, st, K, teacher, L)
        eng.round(slots, K, out_tok, out_cnt, out_done, force=force, dbg=dbg)
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

        draft_flip = False
        want_draft = np.concatenate([[res.a0], res.d_draft])
        for i in range(W):
            if g_draft[i] != want_draft[i]:
                assert res.draft_gap[i] < NEAR_TIE, (
                    f"round {stats.rounds}: draft row {i} gpu {g_draft[i]} oracle {want_draft[i]} "
                    f"gap {res.draft_gap[i]:.4f}")
                stats.near_tie_flips += 1
                draft_flip = True
        if check_logits:
            err = float(np.max(np.abs(dl.cpu().numpy().astype(np.float64) - res.draft_logits)))
            assert err <= logit_tol, f"draft logits err {err}"
            stats.max_logit_err = max(stats.max_logit_err, err)
            stats.logit_rows += W
        # verify rows are compared whenever the verify inputs agree (forcing
        # overwrites draft rows 1..L+1, so a flip there changes no input)
        same_inputs = list(g_vin) == [res.a0] + list(res.d)
        assert same_inputs or draft_flip, (
            f"round {stats.rounds}: verify inputs differ without a draft flip: "
            f"{list(g_vin)} vs {[res.a0] + list(res.d)}")
        A = gpu_accept(g_vin, g_vt, K)
        if same_inputs:
            verify_flip = False
            for i in range(W):
                if g_vt[i] != res.a[i]:
                    assert res.verify_gap[i] < NEAR_TIE, (
                        f"round {stats.rounds}: verify row {i} gpu {g_vt[i]} oracle {res.a[i]} "
                        f"gap {res.verify_gap[i]:.4f}")
                    stats.near_tie_flips += 1
                    verify_flip = True
            if not verify_flip:
                assert A == res.A, (stats.rounds, A, res.A)
            if check_logits:
                err = float(np.max(np.abs(vl.cpu().numpy().astype(np.float64) - res.verify_logits)))
                assert err <= logit_tol, f"verify logits err {err}"
                stats.max_logit_err = max(stats.max_logit_err, err)
                stats.logit_rows += W
        stats.accepted.append((L, res.A, A if same_inputs else None))
        # the GPU's own round is consistent with the acceptance rule
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
            eng.restore(slot, st.n, st.x0, len(st.out), max_new, int(st.done), stats.rounds)
    return st, stats


def resync(eng, slot, prompt, st, max_new, rounds):
    """Give a GPU sequence the oracle's token history after a near-tie
    divergence: prefill prefix + committed tokens (all but the boundary), then
    restore the boundary token, output count and round counter."""
    text = np.concatenate([prompt.text, np.asarray(st.out[:-1], dtype=np.int32)])
    eng.prefill(slot, prompt.vis, text, max_new)
    eng.restore(slot, st.n, st.x0, len(st.out), max_new, int(st.done), rounds)


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
