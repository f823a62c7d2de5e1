"""Planted mistakes in the oracle must be caught by its pins (CPU only).

Each case patches one oracle function with a plausible slip (a dropped term,
a wrong sign or index, a swapped operand) and re-runs the pin that should
catch it; the pin must fail.  Nothing here touches the CUDA path.
"""
import numpy as np
import pytest

from oracle import decode as od
from oracle.model import Decoder, KVCache
from tests import test_oracle_pins as pins


def _micro():
    from synth import make_weights
    w = make_weights(pins.MICRO, seed=0, gain_std=0.1)
    return Decoder(pins.MICRO, w), w


def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    return False


def _draft_boundary_sees_masks(dec, cache, x0, K):
    n = cache.seq_len
    ids = np.array([x0] + [dec.cfg.mask_token_id] * K)
    allowed = np.ones((K + 1, n + K + 1), dtype=bool)          # slip: row 0 not causal
    return dec.forward(dec.embed_tokens(ids), n + np.arange(K + 1), allowed, cache)


def _draft_masks_causal(dec, cache, x0, K):
    n = cache.seq_len
    ids = np.array([x0] + [dec.cfg.mask_token_id] * K)
    slots = n + np.arange(K + 1)
    allowed = np.arange(n + K + 1)[None, :] <= slots[:, None]   # slip: no bidirectional block
    return dec.forward(dec.embed_tokens(ids), slots, allowed, cache)


def _verify_off_by_one(dec, cache, a0, d):
    n = cache.seq_len
    K = len(d)
    ids = np.concatenate([[a0], np.asarray(d, dtype=np.int64)])
    slots = n + 1 + np.arange(K + 1)
    keys = np.arange(n + K + 2)
    allowed = keys[None, :] <= np.minimum(slots + 1, n + K + 1)[:, None]   # slip: sees next token
    return dec.forward(dec.embed_tokens(ids), slots, allowed, cache)


def _accept_one_too_many(d, a):
    A = 0
    for dj, aj in zip(d, a):
        A += 1                                                  # slip: counts the mismatch
        if int(dj) != int(aj):
            break
    return A


def _rope_wrong_sign(self, x, pos):
    hd = self.cfg.head_dim
    half = hd // 2
    inv = self.cfg.rope_theta ** (-np.arange(half) * 2.0 / hd)
    ang = pos[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=-1)   # slip: sign


def _attention_no_scale(self, q, k, v, allowed):
    group = self.cfg.n_heads // self.cfg.n_kv_heads
    out = np.empty_like(q)
    for h in range(self.cfg.n_heads):
        s = q[:, h, :] @ k[:, h // group, :].T                             # slip: no 1/sqrt(hd)
        s = np.where(allowed, s, -np.inf)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        out[:, h, :] = (p / p.sum(axis=1, keepdims=True)) @ v[:, h // group, :]
    return out


def _rmsnorm_no_gain(self, x, gain):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + self.cfg.rms_eps)   # slip


def _truncate_one_short(self, n):
    for layer in range(len(self.k)):
        self.k[layer][n - 1:] = np.nan                              # slip: drops the last kept slot
        self.v[layer][n - 1:] = np.nan
    self.seq_len = n


def _reveal_at_threshold_too(conf, masked, tau):
    above = [j for j in masked if conf[j] >= tau]                 # slip: >= instead of >
    return above if above else [max(masked, key=lambda j: (conf[j], -j))]


def _reveal_only_the_best(conf, masked, tau):
    return [max(masked, key=lambda j: (conf[j], -j))]            # slip: ignores the threshold


def _denoise_unshifted(dec, cache, x0, block):
    n = cache.seq_len
    B = len(block)
    ids = np.array([x0] + [dec.cfg.mask_token_id if t is None else int(t) for t in block])
    logits = dec.forward(dec.embed_tokens(ids), n + np.arange(B + 1), od.draft_allowed(n, B), cache)
    return np.concatenate([logits[1:], logits[:1]])               # slip: position j read from row j


def _cache_write_skipped(dec, cache, x0, block):
    cache.truncate(cache.seq_len + len(block))                   # slip: no causal rewrite


def _refine_feedback_off_by_one(dec, cache, x0, K, tau_d):
    fixed = [None] * (K + 1)
    rec = od.RefinedDraft(0, [], [], [], [])
    logits = None
    while any(t is None for t in fixed):
        logits = od.denoise_forward(dec, cache, x0, fixed[1:K + 1])   # slip: slot n+i carries pred i
        conf = np.max(od.softmax_rows(logits), axis=1)
        tok = od.argmax_rows(logits)
        pick = od.reveal_positions(conf, [i for i in range(K + 1) if fixed[i] is None], tau_d)
        for i in pick:
            fixed[i] = int(tok[i])
        rec.steps += 1
        rec.fixed_per_step.append(pick)
        rec.conf_per_step.append(conf)
        rec.gap_per_step.append(od.top2_gap(logits))
        rec.tok_per_step.append(tok)
    return fixed[0], np.array(fixed[1:], dtype=np.int64), logits, rec


MUTATIONS = [
    ("draft boundary row sees the mask block", od, "draft_forward", _draft_boundary_sees_masks,
     "test_boundary_row_is_the_ar_logit"),
    ("draft mask rows not bidirectional", od, "draft_forward", _draft_masks_causal,
     "test_draft_and_verify_masks_follow_paper"),
    ("verify mask off by one", od, "verify_forward", _verify_off_by_one,
     "test_verify_rows_equal_incremental_ar"),
    ("accept counts the first mismatch", od, "accept_length", _accept_one_too_many,
     "test_forced_acceptance_hits_schedule_and_stays_ar"),
    ("RoPE rotation sign", Decoder, "rope", _rope_wrong_sign, "test_rope_matches_complex_rotation"),
    ("softmax scale dropped", Decoder, "attention", _attention_no_scale, "test_causal_forward_matches_torch"),
    ("RMSNorm gain dropped", Decoder, "rmsnorm", _rmsnorm_no_gain, "test_causal_forward_matches_torch"),
    ("cache truncation one short", KVCache, "truncate", _truncate_one_short, "test_self_spec_equals_greedy_ar"),
    ("reveal at the threshold itself", od, "reveal_positions", _reveal_at_threshold_too,
     "test_reveal_rule_cases"),
    ("reveal ignores the threshold", od, "reveal_positions", _reveal_only_the_best,
     "test_diffusion_first_token_is_ar_and_cache_is_ar"),
    ("block prediction not shifted", od, "denoise_forward", _denoise_unshifted,
     "test_diffusion_first_token_is_ar_and_cache_is_ar"),
    ("block cache write skipped", od, "cache_write_forward", _cache_write_skipped,
     "test_diffusion_first_token_is_ar_and_cache_is_ar"),
    ("refined draft fed back one slot early", od, "refine_draft", _refine_feedback_off_by_one,
     "test_refined_drafting_feeds_fixed_predictions_back_at_their_slots"),
]


@pytest.mark.parametrize("name,owner,attr,patched,pin", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pin_catches_planted_mistake(monkeypatch, name, owner, attr, patched, pin):
    dec, w = _micro()
    monkeypatch.setattr(owner, attr, patched)
    fn = getattr(pins, pin)
    if pin == "test_causal_forward_matches_torch":
        caught = _fails(fn, "micro", (dec, w), (dec, w))
    elif pin == "test_draft_and_verify_masks_follow_paper":
        caught = _fails(fn, (dec, w), monkeypatch)
    elif pin == "test_self_spec_equals_greedy_ar":
        caught = _fails(fn, (dec, w), 3)
    elif pin == "test_reveal_rule_cases":
        caught = _fails(fn)
    elif pin == "test_refined_drafting_feeds_fixed_predictions_back_at_their_slots":
        caught = _fails(fn, (dec, w), monkeypatch)
    else:
        caught = _fails(fn, (dec, w))
    assert caught, f"planted mistake not caught: {name}"
