"""CPU oracle for greedy self-speculative draft/verify decoding (test infrastructure).

This package is test infrastructure, not product code.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline arm may import it.
It shares no code with the CUDA path: it reads the same seeded inputs from
``synth`` and nothing else.

Everything is float64, with the bf16 weights and visual embeddings expanded
exactly.  It follows the paper's decoding procedure (Appendix "Self-Speculative
Decoding and KV-Cache Update", Sec. 4.3 and Fig. "Self-speculative decoding")
step by step, with explicit boolean attention masks and a full softmax.

Stochastic decoding (the standard acceptance-rejection rule the paper names
in Sec. 3, with Philox4x32-10 draws) is in ``oracle/sampling.py``, pinned in
``tests/test_oracle_sampling.py``.

Parity status: every function here is pinned by a ``-m "not gpu"`` test
against something other than itself (brute-force attention, a complex-number
RoPE, closed forms of RMSNorm, a torch fp64 causal reference, and the paper's
AR-equivalence theorem); see ``tests/test_oracle_pins.py``.
"""
from .model import Decoder, KVCache  # noqa: F401
from . import sampling  # noqa: F401
from .decode import (  # noqa: F401
    SeqState, RoundResult, prefill, draft_forward, verify_forward, accept_length,
    self_spec_round, ar_decode, self_spec_decode, forced_drafts, tokens_per_forward,
    reveal_positions, denoise_forward, cache_write_forward, diffusion_block, diffusion_decode,
    refine_draft, self_spec_round_refined, reveal_margin,
)
