"""Shared-parameter decoder of the oracle, float64 (test infrastructure only).

The paper adapts one causal decoder so that the same weights run in two
attention modes (Sec. 4 "AR-to-Diffusion Conversion"): token-level causal
(the AR path, Eq. 1-2) and block-causal with bidirectional attention inside
the current block (block diffusion, Eq. 3).  The paper does not print the
decoder architecture; this oracle takes the reading stated in the design
notes: pre-norm blocks, RMSNorm (eps 1e-6, learned gain), rotate-half RoPE
on all 64 head dimensions at 1-D absolute positions (theta 1e4), grouped-query
attention with scale 1/sqrt(64), SwiGLU FFN, untied input/output embeddings,
no biases.

The one mode-dependent ingredient is the attention mask.  ``Decoder.forward``
takes the rows' absolute slots and an explicit boolean mask over key slots, so
the prefill, draft and verify forwards (oracle/decode.py) state their masks
exactly as the paper words them.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

# Query rows per block of one head's score matrix (bounds the temporaries at
# long prefixes; every row's softmax is still taken over all its keys).
ROW_BLOCK = 2048

from synth import ModelConfig, bf16_bits_to_f32


def _f64(bits: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(bits).astype(np.float64)


class KVCache:
    """Per-layer key/value states indexed by absolute slot.

    ``k[l][slot, kv_head, :]`` holds the RoPE-rotated key of the token at
    ``slot``; ``v`` likewise.  ``seq_len`` counts the slots that hold causal
    states of committed tokens.  Slots at or beyond ``seq_len`` are scratch:
    ``truncate`` overwrites them with NaN so that any later read of a freed
    (rejected) state poisons the result instead of passing silently.
    """

    def __init__(self, cfg: ModelConfig, capacity: int):
        shape = (capacity, cfg.n_kv_heads, cfg.head_dim)
        self.k = [np.full(shape, np.nan) for _ in range(cfg.n_layers)]
        self.v = [np.full(shape, np.nan) for _ in range(cfg.n_layers)]
        self.seq_len = 0
        self.capacity = capacity

    def truncate(self, n: int) -> None:
        """Keep slots [0, n); free the rest (paper: rejected states are discarded)."""
        for layer in range(len(self.k)):
            self.k[layer][n:] = np.nan
            self.v[layer][n:] = np.nan
        self.seq_len = n

    def copy(self) -> "KVCache":
        c = KVCache.__new__(KVCache)
        c.k = [a.copy() for a in self.k]
        c.v = [a.copy() for a in self.v]
        c.seq_len = self.seq_len
        c.capacity = self.capacity
        return c


class Decoder:
    """float64 decoder over bf16-valued weights (from ``synth.make_weights``)."""

    def __init__(self, cfg: ModelConfig, weights: dict):
        self.cfg = cfg
        self.embed = _f64(weights["embed"])
        self.lm_head = _f64(weights["lm_head"])
        self.final_norm = _f64(weights["final_norm"])
        self.layers = []
        for lw in weights["layers"]:
            self.layers.append({name: _f64(lw[name]) for name in
                                ("attn_norm", "w_qkv", "w_o", "ffn_norm", "w_gate_up", "w_down")})

    # ------------------------------------------------------------ pieces
    def rmsnorm(self, x: np.ndarray, gain: np.ndarray) -> np.ndarray:
        """RMSNorm: x / sqrt(mean(x^2) + eps) * gain, over the last axis."""
        ms = np.mean(x * x, axis=-1, keepdims=True)
        return x / np.sqrt(ms + self.cfg.rms_eps) * gain

    def rope(self, x: np.ndarray, pos: np.ndarray) -> np.ndarray:
        """Rotate-half RoPE.  x [rows, heads, hd], pos [rows] absolute positions.

        Pair (i, i + hd/2) is rotated by angle pos * theta^(-2i/hd).
        """
        hd = self.cfg.head_dim
        half = hd // 2
        inv_freq = self.cfg.rope_theta ** (-np.arange(half, dtype=np.float64) * 2.0 / hd)
        ang = pos.astype(np.float64)[:, None] * inv_freq[None, :]          # [rows, half]
        cos = np.cos(ang)[:, None, :]
        sin = np.sin(ang)[:, None, :]
        x1, x2 = x[..., :half], x[..., half:]
        return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)

    def attention(self, q: np.ndarray, k: np.ndarray, v: np.ndarray, allowed: np.ndarray
                  ) -> np.ndarray:
        """Masked softmax attention with grouped KV heads.

        q [rows, Hq, hd]; k, v [keys, Hkv, hd]; allowed [rows, keys] bool.
        Query head h reads KV head h // (Hq / Hkv).  Scores are scaled by
        1/sqrt(hd); disallowed keys get probability 0.
        """
        cfg = self.cfg
        group = cfg.n_heads // cfg.n_kv_heads
        out = np.empty_like(q)
        scale = 1.0 / np.sqrt(cfg.head_dim)

        def one_head(h):
            kh = h // group
            for r0 in range(0, q.shape[0], ROW_BLOCK):
                r1 = min(r0 + ROW_BLOCK, q.shape[0])
                a = allowed[r0:r1]
                s = (q[r0:r1, h, :] @ k[:, kh, :].T) * scale               # [rows, keys]
                s = np.where(a, s, -np.inf)
                s = s - np.max(s, axis=1, keepdims=True)
                p = np.where(a, np.exp(s), 0.0)
                p = p / np.sum(p, axis=1, keepdims=True)
                out[r0:r1, h, :] = p @ v[:, kh, :]

        # heads are independent; numpy releases the GIL inside these array
        # operations, so long prefixes evaluate several heads at once
        workers = min(cfg.n_heads, os.cpu_count() or 1, 8)
        if workers <= 1 or q.shape[0] * k.shape[0] < (1 << 20):
            for h in range(cfg.n_heads):
                one_head(h)
        else:
            with ThreadPoolExecutor(max_workers=workers) as ex:
                list(ex.map(one_head, range(cfg.n_heads)))
        return out

    # ------------------------------------------------------------ forward
    def embed_tokens(self, ids: np.ndarray) -> np.ndarray:
        return self.embed[np.asarray(ids, dtype=np.int64)]

    def forward(self, x: np.ndarray, slots: np.ndarray, allowed: np.ndarray, cache: KVCache,
                return_hidden: bool = False):
        """Run all layers over input rows ``x`` [rows, d] placed at absolute ``slots``.

        At every layer the rows' RoPE-rotated keys and values are first written
        into ``cache`` at ``slots``; then each row attends over cache slots
        ``[0, allowed.shape[1])`` where ``allowed`` is True.  Returns logits
        [rows, V] (and the final normalised hidden rows when asked).
        """
        cfg = self.cfg
        hd, Hq, Hkv = cfg.head_dim, cfg.n_heads, cfg.n_kv_heads
        nk = allowed.shape[1]
        h = np.array(x, dtype=np.float64)
        slots = np.asarray(slots, dtype=np.int64)
        for li, lw in enumerate(self.layers):
            xn = self.rmsnorm(h, lw["attn_norm"])
            qkv = xn @ lw["w_qkv"].T
            q = qkv[:, : Hq * hd].reshape(-1, Hq, hd)
            k = qkv[:, Hq * hd: (Hq + Hkv) * hd].reshape(-1, Hkv, hd)
            v = qkv[:, (Hq + Hkv) * hd:].reshape(-1, Hkv, hd)
            q = self.rope(q, slots)
            k = self.rope(k, slots)
            cache.k[li][slots] = k
            cache.v[li][slots] = v
            o = self.attention(q, cache.k[li][:nk], cache.v[li][:nk], allowed)
            h = h + o.reshape(-1, Hq * hd) @ lw["w_o"].T
            xn = self.rmsnorm(h, lw["ffn_norm"])
            gu = xn @ lw["w_gate_up"].T
            g, u = gu[:, : cfg.d_ffn], gu[:, cfg.d_ffn:]
            act = g / (1.0 + np.exp(-g)) * u                                 # SiLU(g) * u
            h = h + act @ lw["w_down"].T
        hf = self.rmsnorm(h, self.final_norm)
        logits = hf @ self.lm_head.T
        if return_hidden:
            return logits, hf
        return logits
