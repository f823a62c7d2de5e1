"""Seeded input generators: bf16 encoding, determinism, forced-acceptance schedule."""
import numpy as np
import torch

import synth


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * 3,
        np.array([0.0, -0.0, 1.0, 1.00390625, 1.005859375, 65504.0, 1e-30, -2.5e-3], np.float32),
        # exact ties between two bf16 values: round to even
        (np.arange(0x3F800000, 0x3F800000 + 0x10000 * 4, 0x8000, dtype=np.uint32)).view(np.float32),
    ])
    got = synth.f32_to_bf16_bits(x)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)
    back = synth.bf16_bits_to_f32(got)
    np.testing.assert_array_equal(back, torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_generators_are_deterministic_and_independent():
    cfg = synth.TINY
    a = synth.make_weights(cfg, seed=0)
    b = synth.make_weights(cfg, seed=0)
    np.testing.assert_array_equal(a["layers"][1]["w_down"], b["layers"][1]["w_down"])
    assert not np.array_equal(a["embed"], a["lm_head"])
    c = synth.make_weights(cfg.with_(n_layers=1), seed=0)      # per-tensor streams
    np.testing.assert_array_equal(a["layers"][0]["w_qkv"], c["layers"][0]["w_qkv"])
    w = synth.bf16_bits_to_f32(a["layers"][0]["w_gate_up"])
    assert abs(float(w.std()) - 0.02) < 2e-4 and abs(float(w.mean())) < 2e-4
    p = synth.make_prompt(cfg, 448, 64)
    assert p.text.max() <= cfg.vocab - 2 and p.text.min() >= 0      # never the [M] id
    assert p.vis.shape == (448, cfg.d_model)


def test_censored_geometric_closed_form():
    for alpha in (0.3, 0.893, 0.938, 0.99):
        for K in (4, 16, 32):
            brute = sum(alpha ** j for j in range(1, K + 1))
            assert abs(synth.censored_geometric_mean(alpha, K) - brute) < 1e-12


def test_accept_schedule_moments():
    a16 = synth.solve_alpha(9.7, 16)
    assert abs(a16 - 0.938) < 2e-3
    s = synth.accept_schedule("geometric", 16, 64, 40000)
    assert s.min() >= 0 and s.max() <= 16
    assert abs(s.mean() - 9.7) < 0.03                  # standard error ~0.004
    h = synth.accept_schedule("heavy", 32, 64, 40000)
    assert abs(h.mean() - 9.7) < 0.05
    a32 = synth.solve_alpha((9.7 - 0.1 * 32) / 0.8, 32)
    # the censored geometric part adds its own mass at 0 and at K
    assert abs((h == 32).mean() - (0.1 + 0.8 * a32 ** 32)) < 0.005
    assert abs((h == 0).mean() - (0.1 + 0.8 * (1 - a32))) < 0.005
    assert (synth.accept_schedule("full", 8, 2, 3) == 8).all()


def test_workload_shapes():
    wl = synth.WORKLOADS["serve_b32"]
    ps = wl.prompts()
    assert len(ps) == 32
    for p in ps:
        assert 1024 <= p.length <= 6144
        assert abs(p.vis.shape[0] - 0.75 * p.length) <= 0.5
    g = synth.WORKLOADS["glm_b1"].prompts()[0]
    assert g.vis.shape[0] == 1600 and g.text.shape[0] == 448
    assert synth.weight_bytes(synth.GLM) == 876_609_536
