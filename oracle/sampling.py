"""Stochastic self-speculative decoding (oracle, float64; test infrastructure only).

The paper names the standard acceptance-rejection rule of speculative
sampling for stochastic decoding (Sec. 3 "Speculative Decoding": it
preserves the target distribution) and uses greedy decoding in its
experiments.  This module states that rule for the shared-parameter round:

* the draft forward's boundary row is the causal (target) distribution for
  the next position, so a0 is sampled from it and always kept;
* the mask rows give draft distributions q_1..q_K, from which d_1..d_K are
  sampled independently;
* the verify forward gives the target distributions P_1..P_{K+1}
  (P_j = softmax(verify row j-1 / T), the distribution of the token at the
  slot of d_j given a0, d_1..d_{j-1});
* d_j is accepted while r_j < P_j(d_j) / q_j(d_j) (r_j uniform in (0, 1));
  at the first rejection a replacement is sampled from
  max(0, P_j - q_j) / Z; if every draft is accepted, a bonus token is
  sampled from P_{K+1}; the round commits a0, the accepted drafts and that
  token, and the cache keeps the states of x0, a0 and the accepted drafts.

Random numbers.  Every draw comes from Philox4x32-10 (Salmon, Moraes, Dror
and Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC 2011), keyed by
the user's 64-bit seed, with counter (word group, window row, round, stream
<< 24 | sequence slot); a 32-bit word x gives the uniform
(2 * (x >> 9) + 1) * 2^-24, exact in float32 and never 0 or 1.  Token samples
use the Gumbel-max form: argmax_v (log w_v - log(-log u_v)) samples v with
probability proportional to w_v (u_v the uniform of vocabulary entry v, word
v % 4 of word group v // 4).  Streams: 0 the draft samples (a0, d_j), 2 the
acceptance uniforms (word 0 of group 0), 3 the replacement / bonus samples.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, List, Optional, Tuple

import numpy as np

from .decode import (SeqState, argmax_rows, draft_forward, softmax_rows, top2_gap,
                     verify_forward)
from .model import Decoder

M32 = 0xFFFFFFFF
PHILOX_M0, PHILOX_M1 = 0xD2511F53, 0xCD9E8D57     # round multipliers
PHILOX_W0, PHILOX_W1 = 0x9E3779B9, 0xBB67AE85     # key increments (Weyl sequence)
STREAM_DRAFT, STREAM_ACCEPT, STREAM_SAMPLE = 0, 2, 3


def philox4x32_10(ctr: Tuple, key: Tuple) -> Tuple[np.ndarray, ...]:
    """Philox4x32 with 10 rounds.  ctr: four uint32 arrays (or ints), key: two.
    Each round: (hi0, lo0) = M0 * c0, (hi1, lo1) = M1 * c2 as 64-bit products;
    c <- (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); then the key advances by
    the Weyl constants (not after the last round)."""
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & M32 for c in ctr)
    k0, k1 = (np.uint64(int(k) & M32) for k in key)
    for rnd in range(10):
        p0 = np.uint64(PHILOX_M0) * c0
        p1 = np.uint64(PHILOX_M1) * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(M32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(M32)
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0) & np.uint64(M32), lo1, (hi0 ^ c3 ^ k1) & np.uint64(M32), lo0
        if rnd < 9:
            k0 = (k0 + np.uint64(PHILOX_W0)) & np.uint64(M32)
            k1 = (k1 + np.uint64(PHILOX_W1)) & np.uint64(M32)
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def uniform_from_word(x: np.ndarray) -> np.ndarray:
    """(2 * (x >> 9) + 1) * 2^-24: the midpoint of one of 2^23 equal cells of
    (0, 1), exact in float32 (24 significant bits)."""
    top = (np.asarray(x, dtype=np.uint64) >> np.uint64(9)).astype(np.float64)
    return (2.0 * top + 1.0) * 2.0 ** -24


def uniforms(seed: int, slot: int, rnd: int, stream: int, row: int, n: int) -> np.ndarray:
    """n uniforms for vocabulary entries 0..n-1 of one (slot, round, stream, row)."""
    v = np.arange(n, dtype=np.uint64)
    words = philox4x32_10((v // np.uint64(4), row, rnd, (stream << 24) | slot),
                          (seed & M32, (seed >> 32) & M32))
    w = np.stack(words, axis=0)                                    # [4, n]
    return uniform_from_word(w[(v % np.uint64(4)).astype(np.int64), np.arange(n)])


def gumbel_argmax(logw: np.ndarray, u: np.ndarray) -> Tuple[int, float]:
    """argmax_v logw_v - log(-log u_v) (entries with logw = -inf never win),
    ties to the lowest index; also the gap to the runner-up score."""
    score = np.where(np.isfinite(logw), logw - np.log(-np.log(u)), -np.inf)
    i = int(np.argmax(score))
    rest = np.delete(score, i)
    return i, float(score[i] - (np.max(rest) if rest.size else -np.inf))


def speculative_accept(P: np.ndarray, q: np.ndarray, d: np.ndarray, r: np.ndarray,
                       sample: Callable[[int, np.ndarray], int]) -> Tuple[int, int]:
    """The standard acceptance-rejection rule.  P [K+1, V]: target
    distributions of the K draft positions and the one after; q [K, V]: draft
    distributions; d [K]: drafts (d_j sampled from q_j); r [K]: uniforms.
    d_j is accepted while r_j * q_j(d_j) < P_j(d_j) (r_j < P/q); at the first
    rejection j the next token is sample(j, max(0, P_j - q_j)) (unnormalised
    weights), after K acceptances sample(K, P_{K+1}).  Returns (A, token)."""
    K = len(d)
    for j in range(K):
        if r[j] * q[j, d[j]] < P[j, d[j]]:
            continue
        return j, sample(j, np.maximum(P[j] - q[j], 0.0))
    return K, sample(K, P[K])


@dataclasses.dataclass
class StochasticRound:
    a0: int
    d: np.ndarray            # sampled drafts d_1..d_K
    A: int
    token: int               # replacement or bonus token
    committed: List[int]
    draft_logits: np.ndarray
    verify_logits: np.ndarray
    draft_margin: np.ndarray  # Gumbel-score gap of each draft sample [K+1]
    accept_ratio: np.ndarray  # P_j(d_j) / q_j(d_j), j = 1..K
    r: np.ndarray            # acceptance uniforms
    sample_margin: float     # Gumbel-score gap of the replacement / bonus sample


def self_spec_round_stochastic(dec: Decoder, st: SeqState, K: int, temperature: float,
                               seed: int, slot: int, rnd: int) -> StochasticRound:
    """One stochastic self-speculative round at the given temperature;
    updates ``st`` in place.  ``slot`` and ``rnd`` (rounds since the prefill)
    select the random streams."""
    assert not st.done and temperature > 0
    V = dec.cfg.vocab
    cache = st.cache
    n = cache.seq_len
    inv_t = 1.0 / temperature
    dl = draft_forward(dec, cache, st.x0, K)
    samples, margins = [], []
    for i in range(K + 1):
        logw = dl[i] * inv_t
        tok, gap = gumbel_argmax(logw, uniforms(seed, slot, rnd, STREAM_DRAFT, i, V))
        samples.append(tok)
        margins.append(gap)
    a0, d = samples[0], np.array(samples[1:], dtype=np.int64)
    vl = verify_forward(dec, cache, a0, d)
    P = softmax_rows(vl * inv_t)                                   # P_1..P_{K+1}
    q = softmax_rows(dl[1:] * inv_t) if K else np.zeros((0, V))   # q_1..q_K
    r = np.array([uniforms(seed, slot, rnd, STREAM_ACCEPT, j + 1, 1)[0] for j in range(K)])
    gap_box = {}

    def sample(j, w):
        with np.errstate(divide="ignore"):
            logw = np.log(w)
        tok, gap = gumbel_argmax(logw, uniforms(seed, slot, rnd, STREAM_SAMPLE, j + 1, V))
        gap_box["gap"] = gap
        return tok

    A, token = speculative_accept(P, q, d, r, sample)
    run = [a0] + [int(x) for x in d[:A]] + [token]
    committed = []
    for t in run:
        committed.append(t)
        if t == st.eos or len(st.out) + len(committed) >= st.max_new:
            st.done = True
            break
    st.out.extend(committed)
    cache.truncate(n + A + 2)
    st.x0 = token
    ratio = np.array([P[j, d[j]] / q[j, d[j]] for j in range(K)])
    return StochasticRound(a0=a0, d=d, A=A, token=token, committed=committed, draft_logits=dl,
                           verify_logits=vl, draft_margin=np.array(margins), accept_ratio=ratio,
                           r=r, sample_margin=gap_box["gap"])


def ar_sample_decode(dec: Decoder, st: SeqState, temperature: float, seed: int, slot: int
                     ) -> List[int]:
    """Plain AR sampling from the same prefill state (the target process the
    rule preserves in distribution; not the same draws as the rounds)."""
    from .decode import ar_step_forward
    step = 0
    while not st.done:
        logits = ar_step_forward(dec, st.cache, st.x0)[0]
        tok, _ = gumbel_argmax(logits / temperature,
                               uniforms(seed, slot, step, STREAM_DRAFT, 0, dec.cfg.vocab))
        st.x0 = tok
        st.out.append(tok)
        step += 1
        if tok == st.eos or len(st.out) >= st.max_new:
            st.done = True
    return st.out
