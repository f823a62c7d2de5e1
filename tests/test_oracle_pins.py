"""Pins of the CPU oracle against things other than itself (CPU only).

* attention: brute-force softmax in pure-Python loops (math.exp), masks built
  from the paper's row rules as key limits;
* RoPE: the complex-number form and the relative-position property;
* RMSNorm: closed forms;
* the whole causal forward: an independent torch float64 composition
  (F.linear, F.rms_norm, scaled_dot_product_attention with is_causal, complex
  RoPE via torch.polar);
* the round: the paper's AR-equivalence theorem (Appendix "AR-Equivalence and
  Equality Testing"), the boundary logit being the AR logit (Appendix step
  "Draft forward"), verify rows equal to incremental AR logits, commit bounds
  2..K+2, KV-cache contents equal to AR's and no surviving draft state
  (Appendix step "Cache update");
* TPF accounting against the paper's printed tables (tests/golden);
* direct block-diffusion decoding (Appendix "Direct Block-Diffusion
  Decoding"): block size 1 is greedy AR; a threshold above every probability
  reveals one position per step, the most confident; a threshold below every
  probability reveals the block in one step, equal to the one-shot draft; a
  block's first token is the AR prediction; after every block the cache equals
  AR's cache with no bidirectional state left; output cut at the first EOS;
* multi-step drafting (Sec. 6 "Draft Schedule"): committed output equal to
  greedy AR for every threshold, tau_d < 0 is the one-shot round, tau_d > 1
  fixes one prediction per step (the most confident), each fixed prediction
  is fed back at its own slot, and forcing still hits the schedule.
"""
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle import decode as od
from oracle.model import Decoder, KVCache
from synth import TINY, bf16_bits_to_f32, make_prompt, make_weights

HERE = os.path.dirname(os.path.abspath(__file__))

MICRO = TINY.with_(n_layers=2, d_model=128, n_heads=4, n_kv_heads=2, d_ffn=256, vocab=512)


@pytest.fixture(scope="module")
def micro():
    w = make_weights(MICRO, seed=0, gain_std=0.1)
    return Decoder(MICRO, w), w


@pytest.fixture(scope="module")
def tiny():
    w = make_weights(TINY, seed=0, gain_std=0.1)
    return Decoder(TINY, w), w


def _prefill(dec, n_vis=24, n_text=8, max_new=64, eos=-1, cap=256, index=0):
    p = make_prompt(dec.cfg, n_vis, n_text, index=index)
    return od.prefill(dec, p.vis, p.text, cap, max_new, eos)


# ------------------------------------------------------------------ attention
def brute_attention(q, k, v, limits, group):
    """Pure-Python masked softmax: row i attends keys 0..limits[i] inclusive."""
    rows, Hq, hd = q.shape
    out = np.zeros_like(q)
    scale = 1.0 / math.sqrt(hd)
    for i in range(rows):
        for h in range(Hq):
            kh = h // group
            s = []
            for j in range(limits[i] + 1):
                s.append(sum(float(q[i, h, t]) * float(k[j, kh, t]) for t in range(hd)) * scale)
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            for t in range(hd):
                out[i, h, t] = sum(e[j] * float(v[j, kh, t]) for j in range(len(e))) / z
    return out


@pytest.mark.parametrize("mode", ["prefill", "draft", "verify"])
def test_attention_matches_bruteforce(micro, mode):
    dec, _ = micro
    rng = np.random.default_rng(5)
    n, K = 13, 4
    hd, Hq, Hkv = 64, MICRO.n_heads, MICRO.n_kv_heads
    if mode == "prefill":
        rows, nk = n, n
        limits = list(range(n))
        allowed = np.tril(np.ones((n, n), bool))
    elif mode == "draft":
        rows, nk = K + 1, n + K + 1
        limits = [n] + [n + K] * K                   # boundary causal, masks see the window
        keys = np.arange(nk)
        allowed = np.stack([keys <= lim for lim in limits])
    else:
        rows, nk = K + 1, n + K + 2
        limits = [n + 1 + i for i in range(K + 1)]
        keys = np.arange(nk)
        allowed = np.stack([keys <= lim for lim in limits])
    q = rng.standard_normal((rows, Hq, hd))
    k = rng.standard_normal((nk, Hkv, hd))
    v = rng.standard_normal((nk, Hkv, hd))
    got = dec.attention(q, k, v, allowed)
    want = brute_attention(q, k, v, limits, Hq // Hkv)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-12)


def _capture_masks(monkeypatch, dec):
    seen = []
    orig = Decoder.attention

    def spy(self, q, k, v, allowed):
        seen.append(allowed.copy())
        return orig(self, q, k, v, allowed)

    monkeypatch.setattr(Decoder, "attention", spy)
    return seen


def test_draft_and_verify_masks_follow_paper(micro, monkeypatch):
    """Draft: boundary row keys 0..n, mask rows keys 0..n+K.  Verify: row i keys 0..n+1+i."""
    dec, _ = micro
    st = _prefill(dec)
    n, K = st.n, 5
    seen = _capture_masks(monkeypatch, dec)
    od.draft_forward(dec, st.cache, st.x0, K)
    draft_masks = list(seen)
    seen.clear()
    od.verify_forward(dec, st.cache, 7, np.arange(K))
    verify_masks = list(seen)
    assert len(draft_masks) == MICRO.n_layers and len(verify_masks) == MICRO.n_layers
    for m in draft_masks:
        assert m.shape == (K + 1, n + K + 1)
        assert m[0].sum() == n + 1 and m[0, : n + 1].all()
        assert m[1:].all()
    for m in verify_masks:
        assert m.shape == (K + 1, n + K + 2)
        for i in range(K + 1):
            assert m[i].sum() == n + 2 + i and m[i, : n + 2 + i].all()


# ------------------------------------------------------------------ RoPE / RMSNorm
def test_rope_matches_complex_rotation(micro):
    dec, _ = micro
    rng = np.random.default_rng(1)
    x = rng.standard_normal((7, 3, 64))
    pos = np.array([0, 1, 2, 17, 100, 2047, 12321])
    got = dec.rope(x, pos)
    z = x[..., :32] + 1j * x[..., 32:]
    w = 10000.0 ** (-np.arange(32) / 32.0)
    z = z * np.exp(1j * pos[:, None, None] * w[None, None, :])
    want = np.concatenate([z.real, z.imag], axis=-1)
    np.testing.assert_allclose(got, want, atol=1e-12)


def test_rope_relative_and_isometric(micro):
    dec, _ = micro
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 1, 64))
    k = rng.standard_normal((1, 1, 64))
    a = float(np.sum(dec.rope(q, np.array([50])) * dec.rope(k, np.array([20]))))
    b = float(np.sum(dec.rope(q, np.array([1030])) * dec.rope(k, np.array([1000]))))
    assert abs(a - b) < 1e-9
    np.testing.assert_allclose(np.linalg.norm(dec.rope(q, np.array([777]))), np.linalg.norm(q))
    np.testing.assert_allclose(dec.rope(q, np.array([0])), q)


def test_rmsnorm_closed_forms(micro):
    dec, _ = micro
    d = 128
    c = 3.0
    g = np.linspace(0.5, 1.5, d)
    out = dec.rmsnorm(np.full((1, d), c), g)
    np.testing.assert_allclose(out[0], c / math.sqrt(c * c + 1e-6) * g, rtol=1e-14)
    x = np.random.default_rng(3).standard_normal((4, d)) * 7.0
    y = dec.rmsnorm(x, np.ones(d))
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=1)), 1.0, rtol=1e-6)


# ------------------------------------------------------------------ whole forward
def torch_causal_logits(cfg, w, x_rows):
    """Independent float64 torch composition of the causal decoder."""
    def t(bits):
        return torch.from_numpy(bf16_bits_to_f32(bits).astype(np.float64))
    hd, Hq, Hkv = cfg.head_dim, cfg.n_heads, cfg.n_kv_heads
    P = x_rows.shape[0]
    h = torch.from_numpy(x_rows)
    inv = torch.tensor([cfg.rope_theta ** (-2.0 * i / hd) for i in range(hd // 2)], dtype=torch.float64)
    ang = torch.arange(P, dtype=torch.float64)[:, None] * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]          # [P, 1, hd/2]

    def rope(x):                                                       # x [P, H, hd]
        z = torch.complex(x[..., : hd // 2], x[..., hd // 2:]) * rot
        return torch.cat([z.real, z.imag], dim=-1)

    for lw in w["layers"]:
        xn = F.rms_norm(h, (cfg.d_model,), weight=t(lw["attn_norm"]), eps=cfg.rms_eps)
        qkv = F.linear(xn, t(lw["w_qkv"]))
        q = rope(qkv[:, : Hq * hd].reshape(P, Hq, hd))
        k = rope(qkv[:, Hq * hd:(Hq + Hkv) * hd].reshape(P, Hkv, hd))
        v = qkv[:, (Hq + Hkv) * hd:].reshape(P, Hkv, hd)
        k = k.repeat_interleave(Hq // Hkv, dim=1)
        v = v.repeat_interleave(Hq // Hkv, dim=1)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=True)
        h = h + F.linear(o.transpose(0, 1).reshape(P, Hq * hd), t(lw["w_o"]))
        xn = F.rms_norm(h, (cfg.d_model,), weight=t(lw["ffn_norm"]), eps=cfg.rms_eps)
        gate, up = F.linear(xn, t(lw["w_gate_up"])).split(cfg.d_ffn, dim=-1)
        h = h + F.linear(F.silu(gate) * up, t(lw["w_down"]))
    hf = F.rms_norm(h, (cfg.d_model,), weight=t(w["final_norm"]), eps=cfg.rms_eps)
    return F.linear(hf, t(w["lm_head"])).numpy()


@pytest.mark.parametrize("which", ["micro", "tiny"])
def test_causal_forward_matches_torch(which, micro, tiny):
    dec, w = micro if which == "micro" else tiny
    p = make_prompt(dec.cfg, 20, 12, index=3)
    x = np.concatenate([bf16_bits_to_f32(p.vis).astype(np.float64), dec.embed_tokens(p.text)])
    cache = KVCache(dec.cfg, 64)
    slots = np.arange(x.shape[0])
    got = dec.forward(x, slots, slots[None, :] <= slots[:, None], cache)
    want = torch_causal_logits(dec.cfg, w, x)
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-10)


# ------------------------------------------------------------------ the round
@pytest.mark.parametrize("K", [0, 1, 3, 8])
def test_self_spec_equals_greedy_ar(micro, K):
    """Appendix AR-equivalence: under top-1 every committed token is the verifier's argmax."""
    dec, _ = micro
    ar = od.ar_decode(dec, _prefill(dec, max_new=40))
    st = _prefill(dec, max_new=40)
    rounds = od.self_spec_decode(dec, st, K)
    assert st.out == ar
    for r in rounds[:-1]:
        assert 2 <= len(r.committed) <= K + 2


def test_forced_acceptance_hits_schedule_and_stays_ar(micro):
    """With d_1..d_L set to the AR continuation the verifier accepts exactly L."""
    dec, _ = micro
    K, max_new = 6, 60
    ar = od.ar_decode(dec, _prefill(dec, max_new=max_new + K + 4))
    st = _prefill(dec, max_new=max_new)
    P = st.n
    teacher = np.full(P + len(ar) + 1, -1, np.int64)
    teacher[P: P + len(ar)] = ar
    sched = np.array([0, K, 3, 1, K, 2, 5, 0, 4, K, 1, 1, 2, 3, 0, 6, 2, 2, 2, 2, 2, 2])
    rounds = od.self_spec_decode(dec, st, K, teacher=teacher, schedule=sched)
    for i, r in enumerate(rounds[:-1]):
        assert r.A == sched[i]
        assert len(r.committed) == sched[i] + 2
    assert st.out == ar[:max_new]


def test_boundary_row_is_the_ar_logit(micro):
    dec, _ = micro
    st = _prefill(dec)
    c1, c2 = st.cache.copy(), st.cache.copy()
    dl = od.draft_forward(dec, c1, st.x0, 6)
    al = od.ar_step_forward(dec, c2, st.x0)
    np.testing.assert_allclose(dl[0], al[0], rtol=0, atol=1e-10)


def test_verify_rows_equal_incremental_ar(micro):
    dec, _ = micro
    st = _prefill(dec)
    K = 5
    d = np.array([3, 9, 27, 81, 243])
    c_spec = st.cache.copy()
    od.draft_forward(dec, c_spec, st.x0, K)
    vl = od.verify_forward(dec, c_spec, 11, d)
    c_ar = st.cache.copy()
    od.ar_step_forward(dec, c_ar, st.x0)
    for i, tok in enumerate([11] + list(d)):
        al = od.ar_step_forward(dec, c_ar, tok)
        np.testing.assert_allclose(vl[i], al[0], rtol=0, atol=1e-10)


def test_k0_round_is_two_ar_steps(micro):
    dec, _ = micro
    st = _prefill(dec)
    r = od.self_spec_round(dec, st, 0)
    ar = od.ar_decode(dec, _prefill(dec, max_new=3))
    assert r.A == 0 and r.committed == ar[1:3]


def test_cache_matches_ar_and_no_draft_state_survives(micro):
    dec, _ = micro
    K, max_new = 4, 30
    ar_st = _prefill(dec, max_new=max_new)
    od.ar_decode(dec, ar_st)
    st = _prefill(dec, max_new=max_new)
    P = st.n
    teacher = np.full(P + 64, -1, np.int64)
    teacher[P: P + len(ar_st.out)] = ar_st.out
    sched = np.array([2, 4, 0, 3, 1, 4, 2, 2, 2, 2, 2, 2, 2])
    od.self_spec_decode(dec, st, K, teacher=teacher, schedule=sched)
    # the last round may cache states past the output cap; compare what both hold
    n = min(st.n, ar_st.n)
    assert n >= P + max_new - K - 2
    for layer in range(MICRO.n_layers):
        np.testing.assert_allclose(st.cache.k[layer][:n], ar_st.cache.k[layer][:n], atol=1e-10)
        np.testing.assert_allclose(st.cache.v[layer][:n], ar_st.cache.v[layer][:n], atol=1e-10)
        assert np.isnan(st.cache.k[layer][st.n:]).all()


def test_stop_token_truncates_round(micro):
    dec, _ = micro
    ar = od.ar_decode(dec, _prefill(dec, max_new=40))
    eos = ar[13]
    cut = ar.index(eos) + 1
    st = _prefill(dec, max_new=40, eos=eos)
    P = st.n
    teacher = np.full(P + 64, -1, np.int64)
    teacher[P: P + len(ar)] = ar
    od.self_spec_decode(dec, st, 8, teacher=teacher, schedule=np.full(40, 8))
    assert st.out == ar[:cut] and st.done


@pytest.mark.parametrize("max_new", [1, 2, 3, 17])
def test_output_cap(micro, max_new):
    dec, _ = micro
    ar = od.ar_decode(dec, _prefill(dec, max_new=max_new))
    st = _prefill(dec, max_new=max_new)
    od.self_spec_decode(dec, st, 4)
    assert len(st.out) == max_new and st.out == ar


# ------------------------------------------------------------------ TPF accounting
def _golden_rows():
    rows = []
    with open(os.path.join(HERE, "golden", "tpf_tables.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                src, acc, tpf = line.split()
                rows.append((src, float(acc), float(tpf)))
    return rows


@pytest.mark.parametrize("src,accepted,tpf", _golden_rows())
def test_tpf_accounting_matches_paper_tables(src, accepted, tpf):
    """Every round commits A + 2 tokens over 2 forwards (Sec. 5 TPF definition)."""
    n_rounds = 1000
    got = oracle.tokens_per_forward([accepted + 2] * n_rounds)
    assert abs(got - tpf) <= 0.05 + 1e-9, (src, got, tpf)


# ------------------------------------------------------------------ direct block diffusion
def test_reveal_rule_cases():
    """Every masked position above the threshold is revealed (strictly above);
    if none is, the single most confident one, ties to the lowest position."""
    conf = np.array([0.2, 0.9, 0.5, 0.95, 0.5])
    assert od.reveal_positions(conf, [0, 1, 2, 3, 4], 0.8) == [1, 3]
    assert od.reveal_positions(conf, [0, 2, 4], 0.8) == [2]          # none above: the max, lowest
    assert od.reveal_positions(conf, [0, 2, 4], 0.5) == [2]          # 0.5 is not above 0.5
    assert od.reveal_positions(conf, [4], 2.0) == [4]
    assert od.reveal_positions(conf, [0, 1, 2, 3, 4], -1.0) == [0, 1, 2, 3, 4]


@pytest.mark.parametrize("tau", [-1.0, 0.5, 2.0])
def test_diffusion_block_size_one_is_greedy_ar(micro, tau):
    """B = 1: the only prediction comes from the causal boundary row, so direct
    block diffusion emits the greedy AR sequence for any threshold."""
    dec, _ = micro
    ar = od.ar_decode(dec, _prefill(dec, max_new=24))
    st = _prefill(dec, max_new=24)
    blocks = od.diffusion_decode(dec, st, 1, tau)
    assert st.out == ar
    assert all(b.steps == 1 for b in blocks)


def test_diffusion_threshold_above_one_reveals_the_most_confident(micro):
    """No probability exceeds 1.5: each step reveals exactly one position, the
    masked one whose prediction is the most confident (brute force over the
    recorded confidences), so a block takes B steps."""
    dec, _ = micro
    B = 5
    st = _prefill(dec, max_new=1 + 3 * B)
    blocks = od.diffusion_decode(dec, st, B, 1.5)
    assert len(blocks) == 3
    for b in blocks:
        assert b.steps == B
        masked = set(range(1, B + 1))
        for rev, conf in zip(b.revealed_per_step, b.conf_per_step):
            assert len(rev) == 1
            best = max(sorted(masked), key=lambda j: (conf[j - 1], -j))
            assert rev == [best]
            masked.remove(best)


def test_diffusion_threshold_below_zero_is_the_one_shot_draft(micro):
    """Every probability exceeds -1: the block is revealed in one step, and it is
    the self-speculative one-shot draft [a0, d_1..d_{B-1}] of a window of B masks."""
    dec, _ = micro
    B = 6
    st = _prefill(dec, max_new=40)
    c = st.cache.copy()
    tok = od.argmax_rows(od.draft_forward(dec, c, st.x0, B))
    b = od.diffusion_block(dec, st, B, -1.0)
    assert b.steps == 1 and b.block == [int(t) for t in tok[:B]]


def test_diffusion_first_token_is_ar_and_cache_is_ar(micro):
    """The first position of every block is predicted by the causal boundary
    row, so it is the AR prediction after the committed prefix; after every
    block the cache holds exactly AR's causal states of the committed tokens
    (all but the boundary) and nothing beyond them."""
    dec, _ = micro
    B, max_new = 4, 30
    st = _prefill(dec, max_new=max_new)
    conf0 = np.max(od.softmax_rows(od.denoise_forward(dec, st.cache.copy(), st.x0, [None] * B)[:B]),
                   axis=1)
    tau = float(np.median(conf0))       # about half the first step's predictions above
    multi = 0
    while not st.done:
        c = st.cache.copy()
        ar_next = int(od.argmax_rows(od.ar_step_forward(dec, c, st.x0))[0])
        b = od.diffusion_block(dec, st, B, tau)
        assert b.block[0] == ar_next
        multi += any(len(r) > 1 for r in b.revealed_per_step)
        if st.done:
            break
        # AR's cache: the prefix, then one causal step per committed token
        # except the boundary (the last one)
        ref_cache = _prefill(dec, max_new=max_new).cache
        for t in st.out[:-1]:
            od.ar_step_forward(dec, ref_cache, t)
        assert st.n == ref_cache.seq_len
        for layer in range(MICRO.n_layers):
            np.testing.assert_allclose(st.cache.k[layer][:st.n], ref_cache.k[layer][:st.n],
                                       atol=1e-10)
            np.testing.assert_allclose(st.cache.v[layer][:st.n], ref_cache.v[layer][:st.n],
                                       atol=1e-10)
            assert np.isnan(st.cache.k[layer][st.n:]).all()
    assert multi >= 1          # the threshold revealed several positions in one step somewhere


def test_diffusion_stop_token_truncates(micro):
    dec, _ = micro
    B = 4
    st = _prefill(dec, max_new=40)
    od.diffusion_decode(dec, st, B, 0.0)
    free = st.out
    eos = free[9]
    cut = free.index(eos) + 1
    st = _prefill(dec, max_new=40, eos=eos)
    od.diffusion_decode(dec, st, B, 0.0)
    assert st.done and st.out == free[:cut]


# ------------------------------------------------------------------ multi-step drafting
def _median_first_conf(dec, st, K):
    logits = od.denoise_forward(dec, st.cache.copy(), st.x0, [None] * K)
    return float(np.median(np.max(od.softmax_rows(logits), axis=1)))


@pytest.mark.parametrize("tau", [-1.0, "median", 2.0])
def test_refined_drafting_equals_greedy_ar(micro, tau):
    """The verifier decides every committed token, so refining the draft
    changes how many tokens a round commits, never which."""
    dec, _ = micro
    K = 5
    ar = od.ar_decode(dec, _prefill(dec, max_new=36))
    st = _prefill(dec, max_new=36)
    t = _median_first_conf(dec, st, K) if tau == "median" else tau
    while not st.done:
        r, rec = od.self_spec_round_refined(dec, st, K, t)
        assert 1 <= rec.steps <= K + 1
        assert 2 <= len(r.committed) <= K + 2 or st.done
    assert st.out == ar


def test_refined_drafting_below_zero_is_one_shot(micro):
    dec, _ = micro
    K = 6
    a, b = _prefill(dec, max_new=40), _prefill(dec, max_new=40)
    for _ in range(3):
        r1 = od.self_spec_round(dec, a, K)
        r2, rec = od.self_spec_round_refined(dec, b, K, -1.0)
        assert rec.steps == 1
        assert (r1.a0, list(r1.d), list(r1.a), r1.A, r1.committed) == \
            (r2.a0, list(r2.d), list(r2.a), r2.A, r2.committed)
        np.testing.assert_allclose(r1.draft_logits, r2.draft_logits, rtol=0, atol=1e-12)


def test_refined_drafting_above_one_fixes_the_most_confident(micro):
    dec, _ = micro
    K = 4
    st = _prefill(dec, max_new=40)
    _, rec = od.self_spec_round_refined(dec, st, K, 2.0)
    assert rec.steps == K + 1
    open_ = set(range(K + 1))
    for pick, conf in zip(rec.fixed_per_step, rec.conf_per_step):
        best = max(sorted(open_), key=lambda i: (conf[i], -i))
        assert pick == [best]
        open_.remove(best)


def test_refined_drafting_feeds_fixed_predictions_back_at_their_slots(micro, monkeypatch):
    """Prediction i (a0 for i = 0, d_i otherwise) is the token at slot n+1+i:
    once fixed, the next draft forward carries it at that slot instead of [M]
    (prediction K has no slot in the window)."""
    dec, _ = micro
    K = 4
    st = _prefill(dec, max_new=40)
    n = st.n
    windows = []
    real = Decoder.forward

    def spy(self, x, slots, allowed, cache, return_hidden=False):
        ids = [int(np.argmax(np.all(self.embed == row, axis=1))) for row in x]
        windows.append((list(np.asarray(slots)), ids))
        return real(self, x, slots, allowed, cache, return_hidden)

    monkeypatch.setattr(Decoder, "forward", spy)
    _, _, _, rec = od.refine_draft(dec, st.cache.copy(), st.x0, K, 2.0)
    M = MICRO.mask_token_id
    fixed = {}
    assert len(windows) == rec.steps
    for step, (slots, ids) in enumerate(windows):
        assert slots == [n + i for i in range(K + 1)]
        assert ids[0] == st.x0
        for i in range(K):                       # slot n+1+i carries prediction i
            assert ids[1 + i] == fixed.get(i, M), (step, i)
        for i in rec.fixed_per_step[step]:
            fixed[i] = int(rec.tok_per_step[step][i])
    assert sorted(fixed) == list(range(K + 1))


def test_refined_drafting_forced_schedule_hit(micro):
    dec, _ = micro
    K, max_new = 5, 40
    ar = od.ar_decode(dec, _prefill(dec, max_new=max_new + K + 4))
    st = _prefill(dec, max_new=max_new)
    P = st.n
    teacher = np.full(P + len(ar) + 1, -1, np.int64)
    teacher[P:P + len(ar)] = ar
    sched = [0, K, 2, 4, 1, 3, 0, K, 2, 2, 2, 2, 2, 2, 2]
    r = 0
    while not st.done:
        res, _ = od.self_spec_round_refined(dec, st, K, 0.0, teacher, sched[r])
        if not st.done:
            assert res.A == sched[r]
        r += 1
    assert st.out == ar[:max_new]
