"""Pins of the stochastic round in the oracle (CPU only).

* Philox4x32-10 against the known-answer vectors published with the
  generator (Random123's test set: zero counter and key, all-ones, and the
  digits-of-pi counter and key);
* uniforms: the float32-exact map, range and moments;
* the acceptance-rejection rule preserves the target distribution (the
  property the paper cites, Sec. 3 "Speculative Decoding"): on a toy target
  whose next-token distribution depends on the whole prefix and drafts from
  prefix-blind distributions (like the mask rows), the first three output
  tokens (one round, then target sampling up to length 3) follow the target
  joint exactly (chi-square over all 125 outcomes, seeded); three planted
  slips in the rule fail the same test;
* at temperature -> 0 a stochastic round is the greedy round;
* the cache after stochastic rounds is AR's cache over the committed tokens.
"""
import numpy as np
import pytest
from scipy import stats

from oracle import decode as od
from oracle import sampling as sm
from oracle.model import Decoder
from synth import make_prompt, make_weights
from tests.test_oracle_pins import MICRO


def _hex(words):
    return " ".join("%08x" % int(w) for w in words)


def test_philox_known_answers():
    assert _hex(sm.philox4x32_10((0, 0, 0, 0), (0, 0))) == "6627e8d5 e169c58d bc57ac4c 9b00dbd8"
    assert _hex(sm.philox4x32_10((0xFFFFFFFF,) * 4, (0xFFFFFFFF, 0xFFFFFFFF))) == \
        "408f276d 41c83b0e a20bc7c6 6d5451fd"
    assert _hex(sm.philox4x32_10((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344),
                                 (0xA4093822, 0x299F31D0))) == "d16cfe09 94fdcceb 5001e420 24126ea1"
    # vectorised counters give the same words as scalar ones
    v = sm.philox4x32_10((np.arange(5), 7, 9, 11), (3, 4))
    for i in range(5):
        s = sm.philox4x32_10((i, 7, 9, 11), (3, 4))
        assert [int(w[i]) for w in v] == [int(x) for x in s]


def test_uniforms_are_exact_and_uniform():
    u = sm.uniforms(seed=12345, slot=3, rnd=7, stream=0, row=2, n=200000)
    assert u.min() > 0 and u.max() < 1
    assert np.array_equal(u.astype(np.float32).astype(np.float64), u)      # float32-exact
    assert abs(u.mean() - 0.5) < 3e-3 and abs(u.var() - 1 / 12) < 2e-3
    assert not np.array_equal(u[:1000], sm.uniforms(12345, 3, 8, 0, 2, 1000))   # round changes it
    assert np.array_equal(u[:1000], sm.uniforms(12345, 3, 7, 0, 2, 1000))       # deterministic


# ------------------------------------------------------------------ the rule
V_TOY, K_TOY = 5, 2      # K = 2: a bonus token is the third output


class ToyTarget:
    """p(. | prefix) = softmax of a table row chosen by the whole prefix."""

    def __init__(self, seed=0):
        self.rng = np.random.default_rng(seed)
        self.rows = {}

    def p(self, prefix):
        key = tuple(prefix)
        if key not in self.rows:
            z = self.rng.standard_normal(V_TOY) * 1.2
            self.rows[key] = np.exp(z) / np.exp(z).sum()
        return self.rows[key]


def _joint3(target):
    out = np.zeros((V_TOY,) * 3)
    for a in range(V_TOY):
        for b in range(V_TOY):
            for c in range(V_TOY):
                out[a, b, c] = target.p([])[a] * target.p([a])[b] * target.p([a, b])[c]
    return out


def _simulate(rule, n_trials, seed=1):
    target = ToyTarget(0)
    rng = np.random.default_rng(seed)
    q = rng.dirichlet(np.ones(V_TOY) * 0.7, size=K_TOY)
    q[1, 2] = 0.0                                       # a draft that can never propose token 2
    q[1] /= q[1].sum()
    counts = np.zeros((V_TOY,) * 3)
    for _ in range(n_trials):
        d = np.array([rng.choice(V_TOY, p=q[j]) for j in range(K_TOY)])
        P = np.stack([target.p(list(d[:j])) for j in range(K_TOY + 1)])
        r = rng.random(K_TOY)

        def sample(j, w):
            return int(rng.choice(V_TOY, p=w / w.sum()))

        A, tok = rule(P, q, d, r, sample)
        y = [int(x) for x in d[:A]] + [tok]
        while len(y) < 3:
            y.append(int(rng.choice(V_TOY, p=target.p(y))))
        counts[tuple(y[:3])] += 1
    return counts, _joint3(target)


def _chi2_pvalue(counts, probs):
    n = counts.sum()
    exp = probs.ravel() * n
    keep = exp > 0
    chi = float((((counts.ravel() - exp) ** 2)[keep] / exp[keep]).sum())
    return stats.chi2.sf(chi, keep.sum() - 1)


N_TRIALS = 40000


def test_acceptance_rule_preserves_the_target_distribution():
    counts, probs = _simulate(sm.speculative_accept, N_TRIALS)
    assert _chi2_pvalue(counts, probs) > 1e-3


def _accept_inverted(P, q, d, r, sample):
    for j in range(len(d)):
        if r[j] * P[j, d[j]] < q[j, d[j]]:                 # slip: q/P instead of P/q
            continue
        return j, sample(j, np.maximum(P[j] - q[j], 0.0))
    return len(d), sample(len(d), P[len(d)])


def _residual_is_target(P, q, d, r, sample):
    for j in range(len(d)):
        if r[j] * q[j, d[j]] < P[j, d[j]]:
            continue
        return j, sample(j, P[j].copy())                   # slip: P instead of max(0, P - q)
    return len(d), sample(len(d), P[len(d)])


def _bonus_from_draft(P, q, d, r, sample):
    for j in range(len(d)):
        if r[j] * q[j, d[j]] < P[j, d[j]]:
            continue
        return j, sample(j, np.maximum(P[j] - q[j], 0.0))
    return len(d), sample(len(d), q[len(d) - 1].copy())    # slip: bonus from the last draft row


@pytest.mark.parametrize("rule", [_accept_inverted, _residual_is_target, _bonus_from_draft])
def test_planted_rule_mistakes_fail_the_distribution_pin(rule):
    counts, probs = _simulate(rule, N_TRIALS)
    assert _chi2_pvalue(counts, probs) < 1e-6


# ------------------------------------------------------------------ model-level round
@pytest.fixture(scope="module")
def micro():
    w = make_weights(MICRO, seed=0, gain_std=0.1)
    return Decoder(MICRO, w)


def _prefill(dec, max_new=40, index=0):
    p = make_prompt(dec.cfg, 24, 8, index=index)
    return od.prefill(dec, p.vis, p.text, 256, max_new)


def test_zero_temperature_round_is_the_greedy_round(micro):
    """As T -> 0 the Gumbel samples become argmaxes, P_j and q_j one-hot, a draft
    is accepted iff it is the verifier's argmax and the replacement is that
    argmax: the greedy round, token for token."""
    dec = micro
    K = 5
    a, b = _prefill(dec), _prefill(dec)
    for rnd in range(4):
        g = od.self_spec_round(dec, a, K)
        s = sm.self_spec_round_stochastic(dec, b, K, 1e-7, seed=99, slot=0, rnd=rnd)
        assert s.a0 == g.a0 and list(s.d) == list(g.d_draft)
        assert s.A == g.A and s.committed == g.committed and a.n == b.n
        if a.done:
            break


def test_stochastic_rounds_keep_ar_cache_and_commit_bounds(micro):
    dec = micro
    K = 4
    st = _prefill(dec, max_new=30)
    rnd = 0
    while not st.done:
        r = sm.self_spec_round_stochastic(dec, st, K, 1.0, seed=7, slot=2, rnd=rnd)
        assert 0 <= r.A <= K and (len(r.committed) == r.A + 2 or st.done)
        rnd += 1
    ref = _prefill(dec, max_new=30).cache
    for t in st.out[:-1]:
        od.ar_step_forward(dec, ref, t)
    n = min(st.n, ref.seq_len)
    assert n >= 24 + 8 + 30 - K - 2
    for layer in range(MICRO.n_layers):
        np.testing.assert_allclose(st.cache.k[layer][:n], ref.k[layer][:n], atol=1e-10)
        assert np.isnan(st.cache.k[layer][st.n:]).all()


def test_k0_stochastic_round_is_two_ar_samples(micro):
    """K = 0: a0 from the boundary row (stream 0, row 0) and the bonus from the
    verify row (stream 3, row 1): two AR sampling steps with those uniforms."""
    dec = micro
    st = _prefill(dec)
    r = sm.self_spec_round_stochastic(dec, st, 0, 0.8, seed=5, slot=1, rnd=3)
    ar = _prefill(dec)
    l1 = od.ar_step_forward(dec, ar.cache, ar.x0)[0]
    y1, _ = sm.gumbel_argmax(l1 / 0.8, sm.uniforms(5, 1, 3, sm.STREAM_DRAFT, 0, MICRO.vocab))
    l2 = od.ar_step_forward(dec, ar.cache, y1)[0]
    p2 = np.exp(l2 / 0.8 - np.max(l2 / 0.8))
    y2, _ = sm.gumbel_argmax(np.log(p2 / p2.sum()),
                             sm.uniforms(5, 1, 3, sm.STREAM_SAMPLE, 1, MICRO.vocab))
    assert r.A == 0 and r.committed == [y1, y2]
