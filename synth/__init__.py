"""Seeded synthetic inputs for self-speculative draft/verify decoding.

This module is shared by the CPU oracle (``oracle/``) and by the CUDA path's
tests and benchmark.  It holds no arithmetic of the decoding method: no
forward pass, no attention, no argmax and no acceptance rule.  It only defines
the model/workload shapes, draws seeded random numbers, encodes them as bf16
bit patterns and draws the forced-acceptance schedule.

Stand-in for the paper's data: the paper measures on English OmniDocBench
region crops with GravityOCR weights (Sec. 5 setup, Table "decode modes");
neither is available, so every input here is synthetic with the same
structure: a long visual prefix of embeddings followed by prompt tokens, and
accepted draft lengths drawn to the mean the paper reports.

Seeds: weights 0, inputs 1, acceptance schedule 2.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

WEIGHT_SEED = 0
INPUT_SEED = 1
ACCEPT_SEED = 2
WEIGHT_STD = 0.02


# ---------------------------------------------------------------- bf16 codec
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest even); return uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Expand uint16 bf16 bit patterns to float32 (exact)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


# ---------------------------------------------------------------- model shapes
@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Decoder shape.  Pre-norm decoder: RMSNorm -> attention -> RMSNorm -> SwiGLU.

    ``mask_token_id`` is the ``[M]`` row (the one embedding the paper adds to
    the AR model, Sec. 4 "AR-to-Diffusion Conversion"); it is the last
    vocabulary row.  ``eos_token_id`` -1 disables the stop token.
    """
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ffn: int
    vocab: int
    rope_theta: float = 10000.0
    rms_eps: float = 1e-6
    eos_token_id: int = -1

    @property
    def mask_token_id(self) -> int:
        return self.vocab - 1

    @property
    def qkv_dim(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim

    def with_(self, **kw) -> "ModelConfig":
        return dataclasses.replace(self, **kw)


TINY = ModelConfig(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64,
                   d_ffn=1024, vocab=4096)
GLM = ModelConfig(n_layers=24, d_model=1024, n_heads=16, n_kv_heads=8, head_dim=64,
                  d_ffn=4096, vocab=59392)


def weight_bytes(cfg: ModelConfig) -> int:
    """Bytes of bf16 matrix weights one forward streams (all layers + LM head)."""
    per_layer = (cfg.qkv_dim * cfg.d_model + cfg.d_model * cfg.n_heads * cfg.head_dim
                 + 2 * cfg.d_ffn * cfg.d_model + cfg.d_model * cfg.d_ffn)
    return 2 * (cfg.n_layers * per_layer + cfg.vocab * cfg.d_model)


# ---------------------------------------------------------------- weights
def _rng(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed, spawn_key=key)))


def _normal_bf16(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    x = rng.standard_normal(shape, dtype=np.float32)
    x *= np.float32(std)
    return f32_to_bf16_bits(x)


def _gain_bf16(rng: np.random.Generator, d: int, gain_std: float) -> np.ndarray:
    if gain_std == 0.0:
        return f32_to_bf16_bits(np.ones(d, np.float32))
    return f32_to_bf16_bits(1.0 + gain_std * rng.standard_normal(d, dtype=np.float32))


def make_weights(cfg: ModelConfig, seed: int = WEIGHT_SEED, gain_std: float = 0.0
                 ) -> Dict[str, object]:
    """Random-init decoder weights as bf16 bit arrays (uint16).

    Layout (row-major, ``[out_features, in_features]``):
      embed     [V, d]            input embedding, row V-1 is ``[M]``
      lm_head   [V, d]            output embedding (untied)
      final_norm[d]
      layers[i] = {attn_norm [d], w_qkv [(Hq+2Hkv)*hd, d] (q heads, then k, then v),
                   w_o [d, Hq*hd], ffn_norm [d], w_gate_up [2F, d] (gate rows then up rows),
                   w_down [d, F]}
    Matrix entries ~ N(0, 0.02); norm gains 1 (or 1 + N(0, gain_std) when a test
    wants the gains exercised).  Each tensor has its own seed stream, so a
    tensor does not depend on the generation order.
    """
    d, F, V = cfg.d_model, cfg.d_ffn, cfg.vocab
    w: Dict[str, object] = {
        "embed": _normal_bf16(_rng(seed, 0, 0), (V, d), WEIGHT_STD),
        "lm_head": _normal_bf16(_rng(seed, 0, 1), (V, d), WEIGHT_STD),
        "final_norm": _gain_bf16(_rng(seed, 0, 2), d, gain_std),
    }
    layers = []
    for li in range(cfg.n_layers):
        layers.append({
            "attn_norm": _gain_bf16(_rng(seed, 1 + li, 0), d, gain_std),
            "w_qkv": _normal_bf16(_rng(seed, 1 + li, 1), (cfg.qkv_dim, d), WEIGHT_STD),
            "w_o": _normal_bf16(_rng(seed, 1 + li, 2), (d, cfg.n_heads * cfg.head_dim), WEIGHT_STD),
            "ffn_norm": _gain_bf16(_rng(seed, 1 + li, 3), d, gain_std),
            "w_gate_up": _normal_bf16(_rng(seed, 1 + li, 4), (2 * F, d), WEIGHT_STD),
            "w_down": _normal_bf16(_rng(seed, 1 + li, 5), (d, F), WEIGHT_STD),
        })
    w["layers"] = layers
    return w


# ---------------------------------------------------------------- prompts
@dataclasses.dataclass
class Prompt:
    """One document crop: visual prefix embeddings then prompt text tokens."""
    vis: np.ndarray      # uint16 bf16 bits [n_vis, d]
    text: np.ndarray     # int32 [n_text], uniform over [0, V-2] (never [M])

    @property
    def length(self) -> int:
        return int(self.vis.shape[0] + self.text.shape[0])


def make_prompt(cfg: ModelConfig, n_vis: int, n_text: int, seed: int = INPUT_SEED,
                index: int = 0) -> Prompt:
    rng = _rng(seed, 100, index)
    vis = _normal_bf16(rng, (n_vis, cfg.d_model), 1.0)
    text = rng.integers(0, cfg.vocab - 1, size=n_text, dtype=np.int64).astype(np.int32)
    return Prompt(vis=vis, text=text)


# ---------------------------------------------------------------- acceptance schedule
def censored_geometric_mean(alpha: float, K: int) -> float:
    """E[min(G, K)] for P(G >= j) = alpha**j."""
    if alpha == 1.0:
        return float(K)
    return alpha * (1.0 - alpha ** K) / (1.0 - alpha)


def solve_alpha(mean: float, K: int) -> float:
    """Bisection for the alpha whose censored geometric has the given mean."""
    if not (0.0 < mean < K):
        raise ValueError("mean must lie in (0, K)")
    lo, hi = 0.0, 1.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if censored_geometric_mean(mid, K) < mean:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def rounds_used(sched_row: np.ndarray, max_new: int) -> int:
    """Rounds one sequence runs under a forced schedule: every round commits
    L + 2 tokens and the prefill's boundary token is the first output, so
    rounds run until max_new tokens are out (the last one may be cut)."""
    n_out, r = 1, 0
    while n_out < max_new:
        n_out += int(sched_row[r]) + 2
        r += 1
    return r


def realized_mean(sched: np.ndarray, max_new: int) -> float:
    """Mean forced L over the rounds the sequences actually run."""
    used = [sched[i, :rounds_used(sched[i], max_new)] for i in range(sched.shape[0])]
    return float(np.concatenate(used).mean())


def accept_schedule(kind: str, K: int, n_seq: int, n_rounds: int, mean: float = 9.7,
                    seed: int = ACCEPT_SEED, max_new: Optional[int] = None,
                    tol: float = 0.1) -> np.ndarray:
    """Forced accepted-draft lengths L[seq, round], int32 in [0, K].

    kind "geometric": L = min(G, K), P(G >= j) = alpha**j, alpha solved for ``mean``.
    kind "heavy":     10% L = K, 10% L = 0, 80% censored geometric whose mean makes
                      the mixture mean ``mean``.
    kind "full"/"zero": always K / always 0.

    With ``max_new``, the draw is conditioned on the rounds a decode of
    max_new tokens actually runs: draws (numbered 0, 1, ... in the seed key)
    are taken until the mean L over those rounds lies within ``tol`` of
    ``mean``, so a short decode realizes the stated mean.
    """
    if max_new is None or kind in ("full", "zero"):
        return _draw_schedule(kind, K, n_seq, n_rounds, mean, seed, 0)
    for attempt in range(10000):
        s = _draw_schedule(kind, K, n_seq, n_rounds, mean, seed, attempt)
        if abs(realized_mean(s, max_new) - mean) <= tol:
            return s
    raise RuntimeError("no schedule draw realizes the mean within tol")


def _draw_schedule(kind: str, K: int, n_seq: int, n_rounds: int, mean: float, seed: int,
                   attempt: int) -> np.ndarray:
    rng = _rng(seed, 200, K) if attempt == 0 else _rng(seed, 200, K, attempt)
    shape = (n_seq, n_rounds)
    if kind == "full":
        return np.full(shape, K, np.int32)
    if kind == "zero":
        return np.zeros(shape, np.int32)

    def geo(alpha, size):
        u = rng.random(size)
        # G >= j  <=>  u < alpha**j  ; G = floor(log(u)/log(alpha))
        g = np.floor(np.log(np.maximum(u, 1e-300)) / math.log(alpha))
        return np.minimum(g, K).astype(np.int32)

    if kind == "geometric":
        return geo(solve_alpha(mean, K), shape)
    if kind == "heavy":
        inner_mean = (mean - 0.1 * K) / 0.8
        g = geo(solve_alpha(inner_mean, K), shape)
        u = rng.random(shape)
        g = np.where(u < 0.1, K, np.where(u < 0.2, 0, g)).astype(np.int32)
        return g
    raise ValueError(kind)


# ---------------------------------------------------------------- workloads
@dataclasses.dataclass(frozen=True)
class Workload:
    """One benchmark / parity configuration (shapes of the paper's workloads)."""
    name: str
    model: ModelConfig
    batch: int
    prefix_min: int
    prefix_max: int
    vis_frac: float
    K: int
    max_new: int
    accept: str              # "natural" | "geometric" | "heavy"
    accept_mean: float = 9.7
    n_vis_fixed: Optional[int] = None

    def prompts(self, seed: int = INPUT_SEED) -> List[Prompt]:
        rng = _rng(seed, 300)
        out = []
        for i in range(self.batch):
            if self.prefix_min == self.prefix_max:
                P = self.prefix_min
            else:
                P = int(rng.integers(self.prefix_min, self.prefix_max + 1))
            n_vis = self.n_vis_fixed if self.n_vis_fixed is not None else int(round(self.vis_frac * P))
            out.append(make_prompt(self.model, n_vis, P - n_vis, seed, i))
        return out

    def max_rounds(self) -> int:
        # every round commits at least 2 tokens; the prefill commits 1
        return self.max_new // 2 + 1

    def schedule(self, K: Optional[int] = None, mean: Optional[float] = None
                 ) -> Optional[np.ndarray]:
        """Forced L per (sequence, round), drawn so that the rounds a decode of
        max_new tokens runs realize the mean within 0.1 (``accept_schedule``).
        ``K`` and ``mean`` override the workload's block size and mean."""
        if self.accept == "natural":
            return None
        K = self.K if K is None else K
        mean = self.accept_mean if mean is None else mean
        return accept_schedule(self.accept, K, self.batch, self.max_new // 2 + 1, mean,
                               max_new=self.max_new)


WORKLOADS: Dict[str, Workload] = {
    # tiny decoder, natural drafting (no forcing), 64 rounds
    "tiny": Workload("tiny", TINY, 1, 512, 512, 0.875, 8, 129, "natural", n_vis_fixed=448),
    # GLM-OCR-scale decoder, batch 1, prefix 1600 visual + 448 text, K=16, 512 output tokens
    "glm_b1": Workload("glm_b1", GLM, 1, 2048, 2048, 0.78125, 16, 512, "geometric", n_vis_fixed=1600),
    # serving batch: 32 documents, prefix U[1024, 6144], 75% visual, K=16
    "serve_b32": Workload("serve_b32", GLM, 32, 1024, 6144, 0.75, 16, 512, "geometric"),
    # long dense page: batch 8, prefix 8192 (7168 visual), K=32, 4096 output tokens
    "long_b8": Workload("long_b8", GLM, 8, 8192, 8192, 0.875, 32, 4096, "heavy", n_vis_fixed=7168),
}

# attention-only sweep: K x batch x prefix
SWEEP_K = (4, 8, 16, 32, 64)
SWEEP_BATCH = (1, 8, 64)
SWEEP_PREFIX = (1024, 4096, 8192)


def attn_inputs(batch: int, W: int, ctx: int, n_heads: int = 16, n_kv_heads: int = 8,
                head_dim: int = 64, seed: int = INPUT_SEED, index: int = 0):
    """Q [batch, W, Hq, hd] and K/V [batch, ctx, Hkv, hd]: N(0,1) draws rounded
    to fp16 (the attention kernel's operand type), as np.float16 arrays."""
    rng = _rng(seed, 400, index)
    q = rng.standard_normal((batch, W, n_heads, head_dim), dtype=np.float32).astype(np.float16)
    k = rng.standard_normal((batch, ctx, n_kv_heads, head_dim), dtype=np.float32).astype(np.float16)
    v = rng.standard_normal((batch, ctx, n_kv_heads, head_dim), dtype=np.float32).astype(np.float16)
    return q, k, v
