"""Greedy self-speculative decoding and plain greedy AR decoding (oracle, float64).

Test infrastructure only.  Follows the paper's round (Appendix "Self-Speculative
Decoding and KV-Cache Update", steps State / Draft forward / Verify forward /
Accept / Cache update / Next round; Sec. 4.3; Fig. "Self-speculative
decoding"):

* State: the cache holds causal KV states of every committed token except the
  boundary token x0, the last committed one.  The first x0 is the argmax at
  the prefill's last position.
* Draft forward: window [x0, [M] x K] at slots n..n+K.  The boundary row
  attends causally (keys 0..n); every mask row attends to the cache and to the
  whole window (keys 0..n+K).  a0 = argmax of the boundary row, d_j = argmax of
  mask row j (shifted alignment: the prediction for slot p is read from the
  row at slot p-1, Sec. 4.2 and Appendix "Direct Block-Diffusion Decoding").
* Verify forward: [a0, d_1..d_K] at slots n+1..n+K+1, token-level causal
  (row i sees keys 0..n+1+i); it overwrites the draft's states of the mask
  slots.  a_{i+1} = argmax of row i.
* Accept: A = largest j <= K with d_1..d_j == a_1..a_j; commit a0, d_1..d_A,
  a_{A+1}; keep slots 0..n+1+A (seq_len n+A+2); the next boundary is a_{A+1}.
* Stop: the committed run is cut at the first stop token (or at the output
  cap) and the rest of the round is dropped.

Where the paper is silent the design notes fix the reading (architecture,
[M] id = V-1, causal prefix attention, ties broken to the lowest token id,
absolute RoPE positions of mask slots, output cap counting the prefill's x0).
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np

from synth import bf16_bits_to_f32

from .model import Decoder, KVCache


def argmax_rows(logits: np.ndarray) -> np.ndarray:
    """Greedy token per row; ties go to the lowest token id (np.argmax is first-max)."""
    return np.argmax(logits, axis=1).astype(np.int64)


def top2_gap(logits: np.ndarray) -> np.ndarray:
    """Top-1 minus top-2 logit per row (the near-tie margin)."""
    part = np.partition(logits, -2, axis=1)
    return part[:, -1] - part[:, -2]


@dataclasses.dataclass
class SeqState:
    """Decoding state of one sequence between rounds."""
    cache: KVCache
    x0: int                 # boundary token (committed, not yet in the cache)
    out: List[int]          # committed output tokens, x0 included
    max_new: int            # cap on len(out)
    eos: int = -1
    done: bool = False
    prefill_gap: float = float("inf")   # top-2 gap of the row that chose the first x0

    @property
    def n(self) -> int:
        return self.cache.seq_len


@dataclasses.dataclass
class RoundResult:
    a0: int
    d_draft: np.ndarray     # draft argmax d_1..d_K (before any forcing)
    d: np.ndarray           # drafts fed to the verifier (after forcing)
    a: np.ndarray           # verifier predictions a_1..a_{K+1}
    A: int                  # accepted draft length
    committed: List[int]    # tokens this round commits (after stop truncation)
    draft_logits: np.ndarray
    verify_logits: np.ndarray
    draft_gap: np.ndarray   # top-2 gaps of the draft rows [K+1]
    verify_gap: np.ndarray  # top-2 gaps of the verify rows [K+1]


# ------------------------------------------------------------------ prefill
def prefill(dec: Decoder, vis_bits: np.ndarray, text: np.ndarray, capacity: int,
            max_new: int, eos: int = -1) -> SeqState:
    """Causal forward over [visual embeddings; text tokens] at slots 0..P-1.

    The visual rows replace token embeddings at positions 0..n_vis-1.  The
    prefix is causal (the base decoder is a causal AR model, Sec. 3).  The
    first boundary x0 is the argmax at the last prefix position; it is the
    first committed output token (Appendix, step "State").
    """
    vis = bf16_bits_to_f32(vis_bits).astype(np.float64)
    x = np.concatenate([vis, dec.embed_tokens(text)], axis=0)
    P = x.shape[0]
    cache = KVCache(dec.cfg, capacity)
    slots = np.arange(P)
    allowed = slots[None, :] <= slots[:, None]                     # causal
    logits = dec.forward(x, slots, allowed, cache)
    cache.seq_len = P
    x0 = int(argmax_rows(logits[-1:])[0])
    st = SeqState(cache=cache, x0=x0, out=[x0], max_new=max_new, eos=eos,
                  prefill_gap=float(top2_gap(logits[-1:])[0]))
    st.done = (x0 == eos) or (len(st.out) >= max_new)
    return st


# ------------------------------------------------------------------ masks
def draft_allowed(n: int, K: int) -> np.ndarray:
    """Hybrid draft mask over keys 0..n+K: row 0 (boundary, slot n) sees 0..n;
    mask rows 1..K see the cache and the whole window, 0..n+K."""
    keys = np.arange(n + K + 1)
    allowed = np.empty((K + 1, n + K + 1), dtype=bool)
    allowed[0] = keys <= n
    allowed[1:] = True
    return allowed


def verify_allowed(n: int, K: int) -> np.ndarray:
    """Token-level causal verify mask over keys 0..n+K+1: row i (slot n+1+i) sees 0..n+1+i."""
    slots = n + 1 + np.arange(K + 1)
    return np.arange(n + K + 2)[None, :] <= slots[:, None]


# ------------------------------------------------------------------ forwards
def draft_forward(dec: Decoder, cache: KVCache, x0: int, K: int) -> np.ndarray:
    """Draft forward over [x0, [M] x K] at slots n..n+K (hybrid mask).

    Row 0 (boundary) sees keys 0..n; rows 1..K see keys 0..n+K.  Writes the
    window's KV states (x0's causal state at slot n; the mask slots get
    bidirectional states that the verify forward overwrites).  Returns logits
    [K+1, V].
    """
    n = cache.seq_len
    ids = np.array([x0] + [dec.cfg.mask_token_id] * K)
    slots = n + np.arange(K + 1)
    return dec.forward(dec.embed_tokens(ids), slots, draft_allowed(n, K), cache)


def verify_forward(dec: Decoder, cache: KVCache, a0: int, d: np.ndarray) -> np.ndarray:
    """Verify forward over [a0, d_1..d_K] at slots n+1..n+K+1, token-level causal.

    Row i sees keys 0..n+1+i, i.e. the cache, x0 (written by the draft) and
    the verify window up to itself.  Returns logits [K+1, V].
    """
    n = cache.seq_len
    K = len(d)
    ids = np.concatenate([[a0], np.asarray(d, dtype=np.int64)])
    slots = n + 1 + np.arange(K + 1)
    return dec.forward(dec.embed_tokens(ids), slots, verify_allowed(n, K), cache)


def ar_step_forward(dec: Decoder, cache: KVCache, token: int) -> np.ndarray:
    """One plain AR step: feed ``token`` at slot n (keys 0..n). Returns logits [1, V]."""
    n = cache.seq_len
    allowed = np.ones((1, n + 1), dtype=bool)
    logits = dec.forward(dec.embed_tokens([token]), np.array([n]), allowed, cache)
    cache.seq_len = n + 1
    return logits


# ------------------------------------------------------------------ accept
def accept_length(d: np.ndarray, a: np.ndarray) -> int:
    """A = length of the longest prefix with d_j == a_j (1 <= j <= K)."""
    A = 0
    for dj, aj in zip(d, a):
        if int(dj) != int(aj):
            break
        A += 1
    return A


def forced_drafts(d: np.ndarray, teacher: np.ndarray, n: int, L: int, vocab: int) -> np.ndarray:
    """Benchmark hook (not in the paper): force the accepted length to L.

    ``teacher[p]`` is the greedy-AR token at absolute slot p.  Drafts d_j sit at
    slot n+1+j, so d_j := teacher[n+1+j] for j <= L, and d_{L+1} :=
    (teacher[n+2+L] + 1) mod V when L < K, so that the verifier rejects it.
    """
    d = np.array(d, dtype=np.int64)
    K = len(d)
    for j in range(1, min(L, K) + 1):
        d[j - 1] = teacher[n + 1 + j]
    if L < K:
        d[L] = (int(teacher[n + 2 + L]) + 1) % vocab
    return d


# ------------------------------------------------------------------ round
def self_spec_round(dec: Decoder, st: SeqState, K: int, teacher: Optional[np.ndarray] = None,
                    L: Optional[int] = None) -> RoundResult:
    """One greedy self-speculative round; updates ``st`` in place."""
    assert not st.done
    cache = st.cache
    n = cache.seq_len
    dl = draft_forward(dec, cache, st.x0, K)
    tok = argmax_rows(dl)
    return _verify_accept_commit(dec, st, n, K, int(tok[0]), tok[1:].copy(), dl, teacher, L)


def _verify_accept_commit(dec: Decoder, st: SeqState, n: int, K: int, a0: int,
                          d_draft: np.ndarray, dl: np.ndarray, teacher: Optional[np.ndarray],
                          L: Optional[int]) -> RoundResult:
    """Verify forward, acceptance, commit and cache update of a round whose
    draft (a0, d_1..d_K) is given (Appendix steps Verify forward .. Next round)."""
    cache = st.cache
    d = d_draft if teacher is None else forced_drafts(d_draft, teacher, n, L, dec.cfg.vocab)
    vl = verify_forward(dec, cache, a0, d)
    a = argmax_rows(vl)                                    # a_1..a_{K+1}
    A = accept_length(d, a[:K])
    run = [a0] + [int(x) for x in d[:A]] + [int(a[A])]
    # stop condition: cut at the first stop token or at the output cap
    committed = []
    for t in run:
        committed.append(t)
        if t == st.eos or len(st.out) + len(committed) >= st.max_new:
            st.done = True
            break
    st.out.extend(committed)
    # cache update: causal states of x0, a0, d_1..d_A stay (slots n..n+1+A)
    cache.truncate(n + A + 2)
    st.x0 = int(a[A])
    return RoundResult(a0=a0, d_draft=d_draft, d=d, a=a, A=A, committed=committed,
                       draft_logits=dl, verify_logits=vl,
                       draft_gap=top2_gap(dl), verify_gap=top2_gap(vl))


@dataclasses.dataclass
class RefinedDraft:
    steps: int                           # draft forwards
    fixed_per_step: List[List[int]]      # prediction indices (0 = a0, j = d_j) fixed per step
    conf_per_step: List[np.ndarray]      # confidence of every prediction per step
    gap_per_step: List[np.ndarray]       # top-2 logit gap of every prediction row per step
    tok_per_step: List[np.ndarray]       # argmax of every prediction row per step


def refine_draft(dec: Decoder, cache: KVCache, x0: int, K: int, tau_d: float):
    """Multi-step drafting (Sec. 6 "Draft Schedule", Fig. "Multi-step drafting
    versus one-shot drafting"): the draft window [x0, [M] x K] is re-run, and
    at each step the predictions whose confidence exceeds tau_d are fixed; the
    rest are re-drafted.  Prediction i (a0 for i = 0, d_i otherwise) is read
    from row i; a fixed prediction i < K is fed back as the input at its own
    slot n+1+i in place of the mask there (prediction K has no slot in the
    window).  If no open prediction exceeds tau_d, the single most confident
    one is fixed, as in direct block diffusion, so the draft completes in at
    most K+1 forwards.  Returns (a0, d_1..d_K, the last step's logits, record).
    """
    fixed: List[Optional[int]] = [None] * (K + 1)
    rec = RefinedDraft(steps=0, fixed_per_step=[], conf_per_step=[], gap_per_step=[],
                       tok_per_step=[])
    logits = None
    while any(t is None for t in fixed):
        logits = denoise_forward(dec, cache, x0, fixed[:K])
        conf = np.max(softmax_rows(logits), axis=1)
        tok = argmax_rows(logits)
        masked = [i for i in range(K + 1) if fixed[i] is None]
        pick = reveal_positions(conf, masked, tau_d)
        for i in pick:
            fixed[i] = int(tok[i])
        rec.steps += 1
        rec.fixed_per_step.append(pick)
        rec.conf_per_step.append(conf)
        rec.gap_per_step.append(top2_gap(logits))
        rec.tok_per_step.append(tok)
    return fixed[0], np.array(fixed[1:], dtype=np.int64), logits, rec


def self_spec_round_refined(dec: Decoder, st: SeqState, K: int, tau_d: float,
                            teacher: Optional[np.ndarray] = None, L: Optional[int] = None):
    """A self-speculative round whose draft is refined over several denoising
    steps (``refine_draft``), then verified exactly as a one-shot draft.
    Returns (RoundResult, RefinedDraft)."""
    assert not st.done
    n = st.cache.seq_len
    a0, d_draft, dl, rec = refine_draft(dec, st.cache, st.x0, K, tau_d)
    return _verify_accept_commit(dec, st, n, K, a0, d_draft, dl, teacher, L), rec


def self_spec_decode(dec: Decoder, st: SeqState, K: int, teacher: Optional[np.ndarray] = None,
                     schedule: Optional[np.ndarray] = None, max_rounds: int = 1 << 30
                     ) -> List[RoundResult]:
    rounds = []
    while not st.done and len(rounds) < max_rounds:
        L = None if schedule is None else int(schedule[len(rounds)])
        rounds.append(self_spec_round(dec, st, K, teacher, L))
    return rounds


def ar_decode(dec: Decoder, st: SeqState) -> List[int]:
    """Plain greedy AR from the prefill state: one causal step per token (Eq. 1)."""
    while not st.done:
        logits = ar_step_forward(dec, st.cache, st.x0)
        st.x0 = int(argmax_rows(logits)[0])
        st.out.append(st.x0)
        if st.x0 == st.eos or len(st.out) >= st.max_new:
            st.done = True
    return st.out


# ------------------------------------------------------------------ direct block diffusion
def softmax_rows(logits: np.ndarray) -> np.ndarray:
    """Row-wise softmax in float64."""
    z = logits - np.max(logits, axis=1, keepdims=True)
    e = np.exp(z)
    return e / np.sum(e, axis=1, keepdims=True)


def reveal_positions(conf: np.ndarray, masked: List[int], tau: float) -> List[int]:
    """The confidence rule of direct block-diffusion decoding (Appendix "Direct
    Block-Diffusion Decoding"): every still-masked position whose predicted
    token's probability exceeds tau is revealed; if none does, the single most
    confident masked position is (ties to the lowest position)."""
    above = [j for j in masked if conf[j] > tau]
    if above:
        return above
    best = masked[0]
    for j in masked[1:]:
        if conf[j] > conf[best]:
            best = j
    return [best]


def denoise_forward(dec: Decoder, cache: KVCache, x0: int, block: List[Optional[int]]
                    ) -> np.ndarray:
    """One denoising forward over [x0, block] at slots n..n+B.

    ``block[j-1]`` is the token at block position j (slot n+j), or None while
    it is still masked (fed as [M]).  The boundary row (slot n) attends
    causally to the cache (keys 0..n); every block row attends to the cache
    and to the whole window (keys 0..n+B), the same hybrid mask as the
    self-speculative draft.  Under the shifted alignment, the row at slot
    n+j-1 predicts block position j.  Returns logits [B+1, V]; rows 0..B-1
    are the predictions for positions 1..B.
    """
    n = cache.seq_len
    B = len(block)
    mask_id = dec.cfg.mask_token_id
    ids = np.array([x0] + [mask_id if t is None else int(t) for t in block])
    slots = n + np.arange(B + 1)
    return dec.forward(dec.embed_tokens(ids), slots, draft_allowed(n, B), cache)


def cache_write_forward(dec: Decoder, cache: KVCache, x0: int, block: List[int]) -> None:
    """The pass that extends the cache once a block is complete: a causal
    forward over [x0, y_1..y_{B-1}] at slots n..n+B-1 (row i sees keys
    0..n+i).  It only writes causal KV states; no token is read from it.
    The block's last token y_B becomes the next boundary, whose state the
    next block's first denoising forward writes."""
    n = cache.seq_len
    B = len(block)
    ids = np.array([x0] + [int(t) for t in block[:-1]])
    slots = n + np.arange(B)
    allowed = np.arange(n + B)[None, :] <= slots[:, None]
    dec.forward(dec.embed_tokens(ids), slots, allowed, cache)
    cache.truncate(n + B)


@dataclasses.dataclass
class BlockResult:
    block: List[int]            # y_1..y_B as revealed
    committed: List[int]        # tokens this block commits (after stop truncation)
    steps: int                  # denoising forwards (the cache write not counted)
    revealed_per_step: List[List[int]]   # block positions (1-based) revealed per step
    conf_per_step: List[np.ndarray]      # confidence of every position's prediction per step
    tok_per_step: List[np.ndarray]       # argmax prediction of every position per step
    gap_per_step: List[np.ndarray]       # top-2 logit gap of every position's row per step


def diffusion_block(dec: Decoder, st: SeqState, B: int, tau_c: float) -> BlockResult:
    """Decode one block of B tokens by direct block diffusion and commit it.

    State as in self-speculative decoding: the cache holds the causal states
    of every committed token except the boundary x0 (slot n).  The block is
    initialised with B masks at slots n+1..n+B.  Each denoising step runs
    one forward and reveals positions by ``reveal_positions``; revealed
    tokens stay fixed.  Once complete, one cache-write forward extends the
    cache (slots n..n+B-1) and y_B becomes the boundary.  The committed run is
    cut at the first stop token or at the output cap, which ends generation.
    """
    assert not st.done
    cache = st.cache
    block: List[Optional[int]] = [None] * B
    revealed, confs, toks, gaps = [], [], [], []
    while any(t is None for t in block):
        logits = denoise_forward(dec, cache, st.x0, block)
        probs = softmax_rows(logits[:B])
        conf = np.max(probs, axis=1)
        tok = argmax_rows(logits[:B])
        gaps.append(top2_gap(logits[:B]))
        masked = [j for j in range(B) if block[j] is None]
        pick = reveal_positions(conf, masked, tau_c)
        for j in pick:
            block[j] = int(tok[j])
        revealed.append([j + 1 for j in pick])
        confs.append(conf)
        toks.append(tok)
    full = [int(t) for t in block]
    committed = []
    for t in full:
        committed.append(t)
        if t == st.eos or len(st.out) + len(committed) >= st.max_new:
            st.done = True
            break
    st.out.extend(committed)
    if not st.done:
        cache_write_forward(dec, cache, st.x0, full)
        st.x0 = full[-1]
    return BlockResult(block=full, committed=committed, steps=len(revealed),
                       revealed_per_step=revealed, conf_per_step=confs, tok_per_step=toks,
                       gap_per_step=gaps)


def diffusion_decode(dec: Decoder, st: SeqState, B: int, tau_c: float,
                     max_blocks: int = 1 << 30) -> List[BlockResult]:
    """Direct block-diffusion decoding from a prefill state until a stop."""
    out = []
    while not st.done and len(out) < max_blocks:
        out.append(diffusion_block(dec, st, B, tau_c))
    return out


def reveal_margin(conf: np.ndarray, gap: np.ndarray, masked: List[int], picked: List[int],
                  tau: float) -> float:
    """How far one reveal step's decisions are from flipping, in log units:
    the top-2 logit gap of every picked row (its token), the distance of each
    open confidence from the threshold (log scale), and, when the fallback
    picked the single most confident, its log-ratio to the runner-up.  A GPU
    whose logits are within e of these agrees with every decision where the
    margin exceeds 2e."""
    m = float("inf")
    for j in picked:
        m = min(m, float(gap[j]))
    if tau > 0:
        for j in masked:
            m = min(m, abs(math.log(conf[j]) - math.log(tau)))
    if len(picked) == 1 and not any(conf[j] > tau for j in masked) and len(masked) > 1:
        rest = sorted((conf[j] for j in masked if j != picked[0]), reverse=True)
        m = min(m, math.log(conf[picked[0]]) - math.log(rest[0]))
    return m


def tokens_per_forward(committed_per_round: List[int]) -> float:
    """TPF (Sec. 5 "Efficiency Measurement"): committed tokens / forwards, counting
    the draft and the verify forward of every round separately, prefill excluded."""
    if not committed_per_round:
        return 0.0
    return float(sum(committed_per_round)) / (2.0 * len(committed_per_round))
