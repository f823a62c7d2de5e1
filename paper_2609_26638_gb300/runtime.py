"""Device-memory plumbing around libgs: torch owns the weights, workspace and
stream; every computation is a libgs call.

``Engine`` uploads a weight set (bf16 bit arrays, row-major [out, in]) once,
allocates the workspace ``gs_workspace_bytes`` asks for, and forwards
prefill / round / state calls to the C ABI.
"""
from __future__ import annotations

import ctypes
from typing import Optional

import numpy as np
import torch

from . import gs


def bf16_tensor(bits: np.ndarray, device) -> torch.Tensor:
    """uint16 bf16 bit pattern array -> torch.bfloat16 tensor on ``device``."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


class Engine:
    def __init__(self, model, weights: dict, *, max_batch: int, max_ctx: int, max_K: int,
                 max_prefill: int = 4096, split_pages: int = 0, kv_pages: int = 0,
                 device: str = "cuda:0", eos_token_id: Optional[int] = None):
        self.model = model
        self.device = torch.device(device)
        torch.cuda.set_device(self.device)
        self.stream = torch.cuda.Stream(self.device)
        self.max_K = max_K
        self.max_batch = max_batch
        dev = self.device
        self.w = {k: bf16_tensor(weights[k], dev) for k in ("embed", "lm_head", "final_norm")}
        self.layers = [{k: bf16_tensor(v, dev) for k, v in lw.items()} for lw in weights["layers"]]

        c = gs.gs_config()
        c.n_layers, c.d_model = model.n_layers, model.d_model
        c.n_heads, c.n_kv_heads, c.head_dim = model.n_heads, model.n_kv_heads, model.head_dim
        c.d_ffn, c.vocab = model.d_ffn, model.vocab
        c.rope_theta, c.rms_eps = model.rope_theta, model.rms_eps
        c.mask_token_id = model.mask_token_id
        c.eos_token_id = model.eos_token_id if eos_token_id is None else eos_token_id
        c.max_batch, c.max_ctx, c.max_K, c.max_prefill = max_batch, max_ctx, max_K, max_prefill
        c.kv_pages, c.split_pages = kv_pages, split_pages
        self.cfg = c
        self.ws_bytes = gs.gs_workspace_bytes(c)
        if self.ws_bytes == 0:
            raise gs.GsError(gs.GS_ERR_INVALID_ARG, "invalid config")
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device=dev)

        L = model.n_layers
        arr = ctypes.c_void_p * L

        def ptrs(name):
            return arr(*[lw[name].data_ptr() for lw in self.layers])

        self._arrays = {n: ptrs(n) for n in ("attn_norm", "w_qkv", "w_o", "ffn_norm", "w_gate_up",
                                             "w_down")}
        w = gs.gs_weights()
        w.embed = self.w["embed"].data_ptr()
        w.lm_head = self.w["lm_head"].data_ptr()
        w.final_norm = self.w["final_norm"].data_ptr()
        for n, a in self._arrays.items():
            setattr(w, n, ctypes.cast(a, ctypes.POINTER(ctypes.c_void_p)))
        torch.cuda.synchronize(dev)
        self.handle = gs.gs_create(c, w, self.workspace.data_ptr(), self.ws_bytes,
                                   self.stream.cuda_stream)
        self._x0 = torch.zeros(1, dtype=torch.int32, device=dev)

    # ------------------------------------------------------------ calls
    def prefill(self, slot: int, vis_bits: np.ndarray, text: np.ndarray, max_new: int,
                sync: bool = True) -> Optional[int]:
        dev = self.device
        with torch.cuda.stream(self.stream):
            vis = bf16_tensor(vis_bits, dev) if vis_bits is not None and len(vis_bits) else None
            txt = torch.from_numpy(np.ascontiguousarray(text, dtype=np.int32)).to(dev) \
                if text is not None and len(text) else None
        gs.gs_prefill(self.handle, slot, vis.data_ptr() if vis is not None else 0,
                      0 if vis is None else vis.shape[0], txt.data_ptr() if txt is not None else 0,
                      0 if txt is None else txt.shape[0], max_new, self._x0.data_ptr())
        # keep the inputs alive until the stream has consumed them
        self._keep = (vis, txt)
        if sync:
            self.stream.synchronize()
            return int(self._x0.cpu()[0])
        return None

    def round(self, slots: torch.Tensor, K: int, out_tok: torch.Tensor, out_cnt: torch.Tensor,
              out_done: torch.Tensor, force: Optional[gs.gs_force] = None,
              dbg: Optional[gs.gs_debug] = None, rule: int = gs.GS_ACCEPT_GREEDY) -> None:
        gs.gs_round(self.handle, slots.data_ptr(), slots.shape[0], K, rule, force,
                    out_tok.data_ptr(), out_cnt.data_ptr(), out_done.data_ptr(), dbg)

    def set_sampling(self, temperature: float, seed: int) -> None:
        gs.gs_set_sampling(self.handle, temperature, seed)

    def diffusion_block(self, slots: torch.Tensor, B: int, tau_c: float, out_tok: torch.Tensor,
                        out_cnt: torch.Tensor, out_done: torch.Tensor,
                        out_steps: Optional[torch.Tensor] = None) -> None:
        gs.gs_diffusion_block(self.handle, slots.data_ptr(), slots.shape[0], B, tau_c,
                              out_tok.data_ptr(), out_cnt.data_ptr(), out_done.data_ptr(),
                              out_steps.data_ptr() if out_steps is not None else 0)

    def round_refined(self, slots: torch.Tensor, K: int, tau_d: float, out_tok: torch.Tensor,
                      out_cnt: torch.Tensor, out_done: torch.Tensor,
                      force: Optional[gs.gs_force] = None,
                      out_steps: Optional[torch.Tensor] = None) -> None:
        gs.gs_round_refined(self.handle, slots.data_ptr(), slots.shape[0], K, tau_d, force,
                            out_tok.data_ptr(), out_cnt.data_ptr(), out_done.data_ptr(),
                            out_steps.data_ptr() if out_steps is not None else 0)

    def round_profile(self, slots: torch.Tensor, K: int, out_tok: torch.Tensor,
                      out_cnt: torch.Tensor, out_done: torch.Tensor,
                      force: Optional[gs.gs_force] = None) -> list:
        """One round replayed as a graph with an event after every kernel:
        [(kind name, device ms)] per launch (see gs_round_profile)."""
        prof = gs.gs_round_profile(self.handle, slots.data_ptr(), slots.shape[0], K, force,
                                   out_tok.data_ptr(), out_cnt.data_ptr(), out_done.data_ptr())
        return [(gs.KIND_NAMES[k], ms) for k, ms in prof]

    def restore(self, slot: int, seq_len: int, x0: int, n_out: int, max_new: int, done: int = 0,
                rounds: int = 0) -> None:
        gs.gs_seq_restore(self.handle, slot, seq_len, x0, n_out, max_new, done, rounds)

    def state(self, slot: int) -> dict:
        return gs.gs_seq_state(self.handle, slot)

    def check(self) -> None:
        gs.gs_sync_check(self.handle)

    def close(self) -> None:
        if getattr(self, "handle", None) is not None:
            self.stream.synchronize()
            gs.gs_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
